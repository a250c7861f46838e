"""The pins have teeth: plausible mistakes planted in the oracle (on the CPU,
in this process only, through monkeypatch) must each fail at least one of the
pin tests that guard that part.  The mistakes are the kinds a restatement
of the paper could make: a dropped term, a wrong sign, a transposed operand,
an off-by-one index or cap, a wrong tie rule, a wrong rounding mode.

Each entry names the oracle function it replaces, the mistake, and the pins
expected to catch it.  Nothing here touches the library or a GPU."""
import sys

import numpy as np
import pytest

from oracle import fo_oracle as O

import test_oracle_layers as TL          # noqa: E402  (tests/ is on sys.path under pytest)
import test_oracle_network as TN         # noqa: E402
import test_oracle_mobile as TM          # noqa: E402
import test_oracle_sched_agg as TS       # noqa: E402
import test_preproc as TP                # noqa: E402

ORIG = {n: getattr(O, n) for n in dir(O) if not n.startswith("__")}
ORIG_GET = O.TaskScheduler.get
ORIG_AGG = O.Aggregator.aggregate


# --------------------------------------------------------------------------
# mutated pieces (each differs from the oracle in one place)
# --------------------------------------------------------------------------

def conv_flipped(x, w, b, stride, pad):
    return ORIG["conv_fwd"](x, w[:, ::-1, ::-1, :].copy(), b, stride, pad)


def conv_no_bias(x, w, b, stride, pad):
    return ORIG["conv_fwd"](x, w, None, stride, pad)


def conv_bwd_dw_transposed(x, w, dy, stride, pad, need_dx):
    dx, dw, db = ORIG["conv_bwd"](x, w, dy, stride, pad, need_dx)
    return dx, dw.transpose(0, 2, 1, 3).copy(), db


def conv_bwd_dx_sign(x, w, dy, stride, pad, need_dx):
    dx, dw, db = ORIG["conv_bwd"](x, w, dy, stride, pad, need_dx)
    return (None if dx is None else -dx), dw, db


def maxpool_bwd_last_max(x, dy):
    best = x[:, 0::2, 0::2].copy()
    arg = np.zeros(best.shape, np.int64)
    order = ((0, 0), (0, 1), (1, 0), (1, 1))
    for t, (a, b) in enumerate(order[1:], start=1):
        cand = x[:, a::2, b::2]
        upd = cand >= best                     # ties go to the last maximum
        best = np.where(upd, cand, best)
        arg = np.where(upd, t, arg)
    dx = np.zeros_like(x)
    for t, (a, b) in enumerate(order):
        dx[:, a::2, b::2] = np.where(arg == t, dy, 0.0)
    return dx


def relu_bwd_one_at_zero(x, dy):
    return dy * (x >= 0.0)


def affine_bwd_swapped(x, scale, dy):
    dx, dsc, dsh = ORIG["affine_bwd"](x, scale, dy)
    return dx, dsh, dsc


def linear_fwd_bias_sign(x, w, b):
    return ORIG["linear_fwd"](x, w, None if b is None else -b)


def linear_bwd_dw_transposed(x, w, dy, need_dx):
    dx, dw, db = ORIG["linear_bwd"](x, w, dy, need_dx)
    return dx, dw.T.reshape(dw.shape).copy(), db


def layernorm_unbiased(x, gamma, beta):
    mu = x.mean(-1, keepdims=True)
    var = x.var(-1, ddof=1, keepdims=True)
    rstd = 1.0 / np.sqrt(var + O.LN_EPS)
    xhat = (x - mu) * rstd
    return xhat * gamma + beta, (xhat, rstd)


def layernorm_bwd_dropped_term(cache, gamma, dy):
    xhat, rstd = cache
    c = xhat.shape[-1]
    dxhat = dy * gamma
    dx = rstd * (dxhat - dxhat.mean(-1, keepdims=True))
    return dx, (dy * xhat).reshape(-1, c).sum(0), dy.reshape(-1, c).sum(0)


def gelu_tanh(x):
    return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))


def attention_unscaled(qkv, lengths, d, heads):
    q = qkv.copy()
    q[..., :d] *= np.sqrt(d // heads)
    return ORIG["attention_fwd"](q, lengths, d, heads)


def attention_unmasked(qkv, lengths, d, heads):
    return ORIG["attention_fwd"](qkv, np.full(len(lengths), qkv.shape[1]), d, heads)


def attention_bwd_no_rowsum(cache, dout, d, heads):
    q, k, v, p = cache
    B, h, L, dh = q.shape
    do = O._split_heads(dout.reshape(B, L, d), B, L, h, dh)
    dv = p.transpose(0, 1, 3, 2) @ do
    dp = do @ v.transpose(0, 1, 3, 2)
    ds = p * dp
    dq = ds @ k / np.sqrt(dh)
    dk = ds.transpose(0, 1, 3, 2) @ q / np.sqrt(dh)
    merge = lambda t: t.transpose(0, 2, 1, 3).reshape(B, L, d)
    return np.concatenate([merge(dq), merge(dk), merge(dv)], -1).reshape(B, L, 1, 3 * d)


def dwconv_stride2_late(x, w, b, stride, pad):
    """Stride-2 depthwise windows start one pixel late in both directions."""
    if stride == 2:
        x = np.concatenate([x[:, 1:], np.zeros_like(x[:, :1])], 1)
        x = np.concatenate([x[:, :, 1:], np.zeros_like(x[:, :, :1])], 2)
    return ORIG["dwconv_fwd"](x, w, b, stride, pad)


def hswish_bwd_half_slope(x, dy):
    return dy * np.where(x < -3.0, 0.0, np.where(x > 3.0, 1.0, (x + 3.0) / 6.0))


def dwconv_bwd_dx_unflipped(x, w, dy, stride, pad, need_dx):
    """The input gradient correlates with the filter instead of its flip."""
    dx, dw, db = ORIG["dwconv_bwd"](x, w[:, ::-1, ::-1].copy(), dy, stride, pad, need_dx)
    return dx, ORIG["dwconv_bwd"](x, w, dy, stride, pad, False)[1], db


def conv_stride2_late(x, w, b, stride, pad):
    """Stride-2 windows start one pixel late in both directions."""
    if stride == 2:
        x = np.concatenate([x[:, 1:], np.zeros_like(x[:, :1])], 1)
        x = np.concatenate([x[:, :, 1:], np.zeros_like(x[:, :, :1])], 2)
    return ORIG["conv_fwd"](x, w, b, stride, pad)


def maxpool_fwd_average(x):
    return 0.25 * (x[:, 0::2, 0::2] + x[:, 0::2, 1::2] + x[:, 1::2, 0::2] + x[:, 1::2, 1::2])


def affine_shift_first(x, scale, shift):
    return (x + shift) * scale


def avgpool_sum(x):
    return x.sum(axis=(1, 2))


def ce_unstabilised(z, labels):
    B = z.shape[0]
    with np.errstate(over="ignore", invalid="ignore"):
        e = np.exp(z)
        se = e.sum(-1, keepdims=True)
        loss = float(np.mean(np.log(se[:, 0]) - z[np.arange(B), labels]))
        dz = e / se
    dz[np.arange(B), labels] -= 1.0
    return loss, dz / B


def layernorm_eps_on_std(x, gamma, beta):
    mu = x.mean(-1, keepdims=True)
    var = ((x - mu) ** 2).mean(-1, keepdims=True)
    rstd = 1.0 / (np.sqrt(var) + O.LN_EPS)
    xhat = (x - mu) * rstd
    return xhat * gamma + beta, (xhat, rstd)


def gelu_bwd_no_density_term(x, dy):
    return dy * ORIG["gelu_fwd"](x) / np.where(x == 0.0, 1.0, x)


def attention_causal(qkv, lengths, d, heads):
    """Each query also sees only the keys up to its own position."""
    B, L = qkv.shape[0], qkv.shape[1]
    dh = d // heads
    t = qkv.reshape(B, L, 3 * d)
    q = O._split_heads(t[..., :d], B, L, heads, dh)
    k = O._split_heads(t[..., d:2 * d], B, L, heads, dh)
    v = O._split_heads(t[..., 2 * d:], B, L, heads, dh)
    s = q @ k.transpose(0, 1, 3, 2) / np.sqrt(dh)
    valid = np.arange(L)[None, :] < np.asarray(lengths)[:, None]
    keep = valid[:, None, None, :] & (np.arange(L)[None, None, None, :] <= np.arange(L)[None, None, :, None])
    s = np.where(keep, s, -np.inf)
    p = np.exp(s - s.max(-1, keepdims=True))
    p = p / p.sum(-1, keepdims=True)
    out = (p @ v).transpose(0, 2, 1, 3).reshape(B, L, 1, d)
    return out, (q, k, v, p)


def attention_interleaved_heads(qkv, lengths, d, heads):
    """Head h takes channels h, h + heads, h + 2 heads, ... instead of a block."""
    dh = d // heads
    perm = np.array([j * heads + hh for hh in range(heads) for j in range(dh)])
    full = np.concatenate([perm, perm + d, perm + 2 * d])
    out_p, cache = ORIG["attention_fwd"](qkv[..., full], lengths, d, heads)
    out = np.empty_like(out_p)
    out[..., perm] = out_p
    return out, cache


def meanpool_bwd_not_averaged(x, lengths, dy):
    dx = np.zeros_like(x)
    for b in range(x.shape[0]):
        dx[b, :lengths[b], 0, :] = dy[b]
    return dx


def meanpool_over_all(x, lengths):
    return x[:, :, 0, :].mean(1)


def avgpool_bwd_unscaled(x, dy):
    return np.broadcast_to(dy[:, None, None, :], x.shape).copy()


def ce_grad_not_averaged(z, labels):
    loss, dz = ORIG["softmax_ce"](z, labels)
    return loss, dz * z.shape[0]


def ce_loss_summed(z, labels):
    loss, dz = ORIG["softmax_ce"](z, labels)
    return loss * z.shape[0], dz


def sgd_dampened(theta, v, g, lr, mu):
    v = mu * v + (1.0 - mu) * g
    return theta - lr * v, v


def sgd_gradient_step(theta, v, g, lr, mu):
    v = mu * v + g
    return theta - lr * g, v


def agg_alpha_off_by_one(self, theta_d, theta_dk, t_k):
    if t_k < 0 or t_k > self.t:
        return O.ERR_ARG, theta_d
    if self.t - t_k > self.D:
        return O.STALE, theta_d
    alpha = 1.0 / (self.t - t_k + 2)
    self.t += 1
    return O.OK, alpha * np.asarray(theta_dk, np.float64) + (1 - alpha) * np.asarray(theta_d, np.float64)


def agg_weights_swapped(self, theta_d, theta_dk, t_k):
    return ORIG_AGG(self, theta_dk, theta_d, t_k)


def agg_stale_at_d(self, theta_d, theta_dk, t_k):
    if 0 <= t_k <= self.t and self.t - t_k >= self.D:
        return O.STALE, theta_d
    return ORIG_AGG(self, theta_d, theta_dk, t_k)


def get_tie_to_highest(self):
    if self.policy != "counter":
        return ORIG_GET(self)
    cand = [k for k in range(self.K) if self.q[k]]
    if not cand:
        return O.EMPTY, -1, -1
    k = min(cand, key=lambda j: (self.c[j], -j))
    slot = self.q[k].popleft()
    self.c[k] += 1
    self.free.append(slot)
    self.on[k] = True
    if self.blocked:
        self.on[self.blocked.popleft()] = True
    return O.OK, k, slot


def get_argmax(self):
    if self.policy != "counter":
        return ORIG_GET(self)
    cand = [k for k in range(self.K) if self.q[k]]
    if not cand:
        return O.EMPTY, -1, -1
    k = max(cand, key=lambda j: (self.c[j], -j))
    slot = self.q[k].popleft()
    self.c[k] += 1
    self.free.append(slot)
    self.on[k] = True
    if self.blocked:
        self.on[self.blocked.popleft()] = True
    return O.OK, k, slot


def get_lifo_free_list(self):
    st, k, slot = ORIG_GET(self)
    if st == O.OK:
        self.free.pop()
        self.free.appendleft(slot)
    return st, k, slot


def put_cap_off_by_one(self, k):
    if not (0 <= k < self.K) or not self.active[k]:
        return O.ERR_ARG, -1
    total = self.queued()
    if total > self.omega or len(self.q[k]) >= self.depth:
        self.on[k] = False
        if not self.q[k] and k not in self.blocked:
            self.blocked.append(k)
        return O.FULL, -1
    if not self.free:
        self.free.append(self.omega + total)        # would-be extra slot beyond the cap
    slot = self.free.popleft()
    self.q[k].append(slot)
    if self.policy == "fifo":
        self.arrivals.append(k)
    if k in self.blocked:
        self.blocked.remove(k)
    self.on[k] = (total + 1 < self.omega) and (len(self.q[k]) < self.depth)
    return O.OK, slot


def bf16_truncate(x):
    x = np.asarray(x, np.float64)
    m, e = np.frexp(x)
    return np.ldexp(np.trunc(np.ldexp(m, 8)), e - 8)


def bf16_ties_away(x):
    x = np.asarray(x, np.float64)
    m, e = np.frexp(x)
    t = np.ldexp(m, 8)
    return np.ldexp(np.sign(t) * np.floor(np.abs(t) + 0.5), e - 8)


def dwconv_flipped(x, w, b, stride, pad):
    return ORIG["dwconv_fwd"](x, w[:, ::-1, ::-1].copy(), b, stride, pad)


def dwconv_bwd_dw_transposed(x, w, dy, stride, pad, need_dx):
    dx, dw, db = ORIG["dwconv_bwd"](x, w, dy, stride, pad, need_dx)
    return dx, dw.transpose(0, 2, 1).copy(), db


def hswish_clip_at_3(x):
    return x * np.clip(x + 3.0, 0.0, 3.0) / 6.0


def hsigmoid_bwd_third(x, dy):
    return dy * np.where((x > -3.0) & (x < 3.0), 1.0 / 3.0, 0.0)


def chmul_bwd_mean(x, s, dy):
    return dy * s[:, None, None, :], (dy * x).mean(axis=(1, 2))


def split_sum_not_max(Oflop, S, b, o, allowed=None):
    L, K = len(Oflop), len(b)
    best_l, best_cost = None, None
    for l in range(1, L + 1):
        if allowed is not None and not allowed[l - 1]:
            continue
        worst = 0.0
        for k in range(K):
            t = sum(float(Oflop[i]) for i in range(l)) / float(o[k]) + float(S[l - 1]) / float(b[k])
            worst = max(worst, t)
        if best_cost is None or worst < best_cost:
            best_l, best_cost = l, worst
    return best_l, best_cost


def split_fastest_device(Oflop, S, b, o, allowed=None):
    L, K = len(Oflop), len(b)
    best_l, best_cost = None, None
    for l in range(1, L + 1):
        if allowed is not None and not allowed[l - 1]:
            continue
        costs = [max(sum(float(Oflop[i]) for i in range(l)) / float(o[k]), float(S[l - 1]) / float(b[k]))
                 for k in range(K)]
        worst = min(costs)
        if best_cost is None or worst < best_cost:
            best_l, best_cost = l, worst
    return best_l, best_cost


def source_mutant(fn, old, new):
    """`fn` with one expression of its source replaced, compiled against
    the oracle's own globals (for mistakes inside the network wiring)."""
    import inspect
    import textwrap
    src = textwrap.dedent(inspect.getsource(fn))
    assert src.count(old) == 1, old
    scope = dict(vars(O))
    exec(compile(src.replace(old, new), f"<mutant of {fn.__name__}>", "exec"), scope)
    return scope[fn.__name__]


backward_residual_dropped = source_mutant(O.backward, 'acc(op["in1"], dy)', "None")
backward_overwrites = source_mutant(O.backward, "G[tid] = rnd(G[tid] + g) if tid in G else rnd(g)", "G[tid] = rnd(g)")
param_shapes_bias_first = source_mutant(
    O.param_shapes,
    """            out.append((i, "W", (op["cout"], op["k"], op["k"], op["cin"])))
            if op["bias"]:
                out.append((i, "b", (op["cout"],)))""",
    """            if op["bias"]:
                out.append((i, "b", (op["cout"],)))
            out.append((i, "W", (op["cout"], op["k"], op["k"], op["cin"])))""")
server_trains_highest_slot = source_mutant(O.Server.step, "self.slots.pop(slot)", "self.slots.pop(max(self.slots))")
rejoin_keeps_counter = source_mutant(O.TaskScheduler.set_active, "self.c[k] = max(self.c[k], min(others))", "pass")
fifo_serves_newest = source_mutant(O.TaskScheduler.get, "k = self.arrivals.popleft()", "k = self.arrivals.pop()")
refused_never_blocked = source_mutant(O.TaskScheduler.put, "self.blocked.append(k)", "pass")
sender_on_at_cap = source_mutant(O.TaskScheduler.put, "(total + 1 < self.omega)", "(total + 1 <= self.omega)")
split_ignores_allowed = source_mutant(O.split_point, "if allowed is not None and not allowed[l - 1]:", "if False:")
split_ties_to_largest = source_mutant(O.split_point, "if best_cost is None or worst < best_cost:",
                                      "if best_cost is None or worst <= best_cost:")
head_weights_rounded = source_mutant(O._weights, 'if storage == "bf16" and i < len(ops) - 1:', 'if storage == "bf16":')
hswish_bwd_open_interval = source_mutant(O.hswish_bwd, "np.where(x < -3.0, 0.0, np.where(x > 3.0, 1.0,",
                                         "np.where(x <= -3.0, 0.0, np.where(x >= 3.0, 1.0,")
hsigmoid_bwd_closed_interval = source_mutant(O.hsigmoid_bwd, "(x > -3.0) & (x < 3.0)", "(x >= -3.0) & (x <= 3.0)")
depth_off_by_one = source_mutant(O.TaskScheduler.put, "len(self.q[k]) >= self.depth", "len(self.q[k]) > self.depth")
future_version_accepted = source_mutant(O.Aggregator.aggregate, "if t_k < 0 or t_k > self.t:", "if t_k < 0:")


def get_empty_argmin_serves_nothing(self):
    """The argmin taken over every device, empty queues included: when the
    least-served device has nothing queued the step does nothing."""
    if self.policy != "counter":
        return ORIG_GET(self)
    k = min(range(self.K), key=lambda j: (self.c[j], j))
    if not self.q[k]:
        return O.EMPTY, -1, -1
    return ORIG_GET(self)


forward_flatten_nchw = source_mutant(O.forward, "y = a.reshape(a.shape[0], -1)",
                                     "y = a.transpose(0, 3, 1, 2).reshape(a.shape[0], -1)")


# --------------------------------------------------------------------------
# the table: mistake -> (patches, pins expected to catch it)
# --------------------------------------------------------------------------

def golden_split_cases():
    return [(TP.test_hand_worked_example, (c,)) for c in TP.GOLD["cases"]]


MUTATIONS = {
    "conv forward: kernel flipped": (
        {"conv_fwd": conv_flipped},
        [(TL.test_conv_fwd_matches_brute_force, (3, 1)), (TL.test_conv_single_channel_is_scipy_correlate, ())]),
    "conv forward: bias dropped": (
        {"conv_fwd": conv_no_bias}, [(TL.test_conv_fwd_matches_brute_force, (3, 1))]),
    "conv backward: weight gradient taps transposed": (
        {"conv_bwd": conv_bwd_dw_transposed}, [(TL.test_conv_bwd_finite_differences, (3, 1))]),
    "conv backward: input gradient sign": (
        {"conv_bwd": conv_bwd_dx_sign}, [(TL.test_conv_bwd_finite_differences, (3, 2))]),
    "max-pool backward: ties to the last maximum": (
        {"maxpool2_bwd": maxpool_bwd_last_max}, [(TL.test_maxpool_tie_goes_to_first_in_row_major_order, ())]),
    "ReLU derivative 1 at zero": (
        {"relu_bwd": relu_bwd_one_at_zero}, [(TL.test_relu_derivative_at_zero_is_zero, ())]),
    "affine backward: scale and shift gradients swapped": (
        {"affine_bwd": affine_bwd_swapped}, [(TL.test_affine_and_linear_fd, ())]),
    "linear forward: bias sign": (
        {"linear_fwd": linear_fwd_bias_sign}, [(TL.test_affine_and_linear_fd, ())]),
    "linear backward: weight gradient transposed": (
        {"linear_bwd": linear_bwd_dw_transposed}, [(TL.test_affine_and_linear_fd, ())]),
    "layernorm: unbiased variance": (
        {"layernorm_fwd": layernorm_unbiased}, [(TL.test_layernorm_invariants_and_fd, ())]),
    "layernorm backward: projection term dropped": (
        {"layernorm_bwd": layernorm_bwd_dropped_term}, [(TL.test_layernorm_invariants_and_fd, ())]),
    "GELU: tanh approximation instead of erf": (
        {"gelu_fwd": gelu_tanh}, [(TL.test_gelu_values_and_fd, ())]),
    "attention: 1/sqrt(d_h) scale dropped": (
        {"attention_fwd": attention_unscaled}, [(TL.test_attention_brute_force_one_row, ())]),
    "attention: key mask ignored": (
        {"attention_fwd": attention_unmasked}, [(TL.test_attention_special_cases, ())]),
    "attention backward: softmax row-sum term dropped": (
        {"attention_bwd": attention_bwd_no_rowsum}, [(TL.test_attention_fd, ())]),
    "depthwise conv: stride-2 windows one pixel late": (
        {"dwconv_fwd": dwconv_stride2_late}, [(TM.test_depthwise_is_a_block_diagonal_convolution, (3, 2))]),
    "depthwise conv backward: input gradient through the unflipped filter": (
        {"dwconv_bwd": dwconv_bwd_dx_unflipped}, [(TM.test_depthwise_is_a_block_diagonal_convolution, (3, 1))]),
    "hard swish derivative (x + 3) / 6 between the kinks": (
        {"hswish_bwd": hswish_bwd_half_slope}, [(TM.test_hard_swish_and_sigmoid_values, ())]),
    "conv forward: stride-2 windows one pixel late": (
        {"conv_fwd": conv_stride2_late}, [(TL.test_conv_fwd_matches_brute_force, (3, 2))]),
    "max-pool forward: the window average instead of its maximum": (
        {"maxpool2_fwd": maxpool_fwd_average}, [(TL.test_maxpool_brute_force_and_fd, ())]),
    "affine forward: shift added before the scale": (
        {"affine_fwd": affine_shift_first}, [(TL.test_affine_and_linear_fd, ())]),
    "average pool forward: the sum, not the mean": (
        {"avgpool_fwd": avgpool_sum}, [(TL.test_avgpool_and_flatten, ())]),
    "cross-entropy: softmax without subtracting the row maximum": (
        {"softmax_ce": ce_unstabilised}, [(TL.test_ce_fd_and_shift_invariance, ())]),
    "layernorm: eps added to the standard deviation": (
        {"layernorm_fwd": layernorm_eps_on_std}, [(TL.test_layernorm_invariants_and_fd, ())]),
    "GELU backward: the x phi(x) term dropped": (
        {"gelu_bwd": gelu_bwd_no_density_term}, [(TL.test_gelu_values_and_fd, ())]),
    "attention: a causal mask on top of the key mask": (
        {"attention_fwd": attention_causal}, [(TL.test_attention_special_cases, ())]),
    "attention: heads take interleaved channels": (
        {"attention_fwd": attention_interleaved_heads}, [(TL.test_attention_brute_force_one_row, ())]),
    "mean-pool backward: not divided by the length": (
        {"meanpool_bwd": meanpool_bwd_not_averaged}, [(TL.test_meanpool, ())]),
    "mean-pool over padded tokens": (
        {"meanpool_fwd": meanpool_over_all}, [(TL.test_meanpool, ())]),
    "average-pool backward: 1/(H W) dropped": (
        {"avgpool_bwd": avgpool_bwd_unscaled}, [(TL.test_avgpool_and_flatten, ())]),
    "cross-entropy gradient not averaged over the batch": (
        {"softmax_ce": ce_grad_not_averaged},
        [(TL.test_ce_zero_logits_closed_form, ()), (TL.test_ce_fd_and_shift_invariance, ())]),
    "cross-entropy loss summed, not averaged": (
        {"softmax_ce": ce_loss_summed}, [(TL.test_ce_zero_logits_closed_form, ())]),
    "SGD momentum with dampening": (
        {"sgd_momentum": sgd_dampened}, [(TL.test_sgd_momentum_constant_gradient_closed_form, ())]),
    "SGD step by the gradient, not the momentum": (
        {"sgd_momentum": sgd_gradient_step}, [(TL.test_sgd_momentum_constant_gradient_closed_form, ())]),
    "bf16 rounding by truncation": (
        {"to_bf16": bf16_truncate}, [(TL.test_to_bf16_ties_to_even, ()), (TL.test_to_bf16_matches_bit_rounding_and_torch, ())]),
    "bf16 rounding ties away from zero": (
        {"to_bf16": bf16_ties_away}, [(TL.test_to_bf16_ties_to_even, ())]),
    "depthwise conv: kernel flipped": (
        {"dwconv_fwd": dwconv_flipped}, [(TM.test_depthwise_is_a_block_diagonal_convolution, (3, 1))]),
    "depthwise conv backward: weight gradient taps transposed": (
        {"dwconv_bwd": dwconv_bwd_dw_transposed}, [(TM.test_depthwise_is_a_block_diagonal_convolution, (3, 2))]),
    "hard swish: ReLU6 clipped at 3": (
        {"hswish_fwd": hswish_clip_at_3}, [(TM.test_hard_swish_and_sigmoid_values, ())]),
    "hard sigmoid derivative 1/3": (
        {"hsigmoid_bwd": hsigmoid_bwd_third}, [(TM.test_hard_swish_and_sigmoid_values, ())]),
    "channel scaling backward: mean instead of sum": (
        {"chmul_bwd": chmul_bwd_mean}, [(TM.test_channel_scaling_gradients, ())]),
    "FedAsync: alpha = 1/(t - t_k + 2)": (
        {"Aggregator.aggregate": agg_alpha_off_by_one},
        [(TS.test_fedasync_matches_hand_worked_golden, ()), (TS.test_running_mean_closed_form, ())]),
    "FedAsync: global and local weights swapped": (
        {"Aggregator.aggregate": agg_weights_swapped},
        [(TS.test_fedasync_matches_hand_worked_golden, ()), (TS.test_running_mean_closed_form, ())]),
    "FedAsync: stale already at t - t_k = D": (
        {"Aggregator.aggregate": agg_stale_at_d},
        [(TS.test_fedasync_matches_hand_worked_golden, ()), (TS.test_running_mean_closed_form, ())]),
    "scheduler: argmin ties to the highest device index": (
        {"TaskScheduler.get": get_tie_to_highest},
        [(TS.test_tiny_schedule_matches_hand_derived_golden, ()), (TS.test_backlogged_queues_are_served_round_robin, ())]),
    "scheduler: argmax instead of argmin": (
        {"TaskScheduler.get": get_argmax}, [(TS.test_tiny_schedule_matches_hand_derived_golden, ())]),
    "scheduler: freed slots reused last-in first-out": (
        {"TaskScheduler.get": get_lifo_free_list},
        [(TS.test_tiny_schedule_matches_hand_derived_golden, ()), (TS.test_slot_reuse_matches_hand_derived_golden, ())]),
    "flow control: cap omega off by one": (
        {"TaskScheduler.put": put_cap_off_by_one},
        [(TS.test_tiny_schedule_matches_hand_derived_golden, ())]
        + [(TS.test_random_traces_keep_invariants_and_pick_min_counter, (s,)) for s in range(4)]),
    "network backward: the residual branch gets no gradient": (
        {"backward": backward_residual_dropped},
        [(TN.test_network_matches_torch_autograd, ("resnet",)), (TN.test_network_finite_differences, ("resnet",))]),
    "network backward: a second gradient contribution overwrites the first": (
        {"backward": backward_overwrites},
        [(TN.test_network_matches_torch_autograd, ("resnet",)), (TN.test_network_matches_torch_autograd, ("mobilenet",))]),
    "network forward: flatten in channel-first order": (
        {"forward": forward_flatten_nchw}, [(TN.test_network_matches_torch_autograd, ("vgg",))]),
    "join: a rejoining device keeps its stale counter": (
        {"TaskScheduler.set_active": rejoin_keeps_counter},
        [(TS.test_leave_drains_queue_and_join_does_not_monopolise, ())]),
    "FIFO policy: newest upload served first": (
        {"TaskScheduler.get": fifo_serves_newest}, [(TS.test_fifo_policy_serves_in_arrival_order, ())]),
    "flow control: a device refused with an empty queue is never turned on again": (
        {"TaskScheduler.put": refused_never_blocked},
        [(TS.test_blocked_device_is_turned_on_by_next_dequeue, ()), (TS.test_slot_reuse_matches_hand_derived_golden, ())]),
    "flow control: Sender left on when the upload reaches the cap": (
        {"TaskScheduler.put": sender_on_at_cap},
        [(TS.test_tiny_schedule_matches_hand_derived_golden, ()), (TS.test_slot_reuse_matches_hand_derived_golden, ())]),
    "bf16 reading: the classifier's weights rounded too": (
        {"_weights": head_weights_rounded}, [(TL.test_bf16_reading_keeps_the_classifier_weights_fp32, ())]),
    "hard swish derivative on the open interval at the kinks": (
        {"hswish_bwd": hswish_bwd_open_interval}, [(TM.test_kink_derivatives_are_the_stated_one_sided_limits, ())]),
    "hard sigmoid derivative 1/6 at the kinks too": (
        {"hsigmoid_bwd": hsigmoid_bwd_closed_interval},
        [(TM.test_kink_derivatives_are_the_stated_one_sided_limits, ())]),
    "flow control: ring depth off by one": (
        {"TaskScheduler.put": depth_off_by_one}, [(TS.test_slot_reuse_matches_hand_derived_golden, ())]),
    "scheduler: empty queues compete in the argmin": (
        {"TaskScheduler.get": get_empty_argmin_serves_nothing},
        [(TS.test_random_traces_keep_invariants_and_pick_min_counter, (s,)) for s in range(4)]),
    "FedAsync: a version from the future accepted": (
        {"Aggregator.aggregate": future_version_accepted}, [(TS.test_stale_and_invalid_versions, ())]),
    "flat layout: conv bias before its weights": (
        {"param_shapes": param_shapes_bias_first}, [(TN.test_flat_layout_is_the_documented_order, ())]),
    "event replay: a step trains on the highest-numbered slot, not the served one": (
        {"Server.step": server_trains_highest_slot}, [(TN.test_server_trains_on_the_batch_the_scheduler_served, ())]),
    "split selection: training and transfer added, not overlapped": (
        {"split_point": split_sum_not_max}, golden_split_cases()),
    "split selection: the allowed split points ignored": (
        {"split_point": split_ignores_allowed}, golden_split_cases()),
    "split selection: ties to the largest l": (
        {"split_point": split_ties_to_largest},
        golden_split_cases() + [(TP.test_ties_go_to_the_smallest_split, ())]),
    "split selection: the fastest device decides": (
        {"split_point": split_fastest_device}, golden_split_cases() + [(TP.test_slowest_device_decides, ())]),
}


def apply(monkeypatch, patches):
    # test_preproc loads the oracle as a top-level module of its own: patch both
    mods = [O] + [m for m in (sys.modules.get("fo_oracle"), TP.O) if m is not None and m is not O]
    for name, fn in patches.items():
        for m in mods:
            if "." in name:
                cls, meth = name.split(".")
                monkeypatch.setattr(getattr(m, cls), meth, fn)
            else:
                monkeypatch.setattr(m, name, fn)


@pytest.mark.parametrize("name", list(MUTATIONS))
def test_planted_mistake_fails_a_pin(name, monkeypatch):
    patches, pins = MUTATIONS[name]
    apply(monkeypatch, patches)
    caught = []
    for fn, args in pins:
        try:
            fn(*args)
        except Exception:           # a failed assertion, or a pin the mistake crashes
            caught.append(fn.__name__)
    assert caught, f"no pin caught the planted mistake: {name}"


def test_unmutated_pins_pass():
    """The same pin calls pass on the oracle as written (so a catch above is
    the planted mistake, not a broken pin)."""
    seen = set()
    for _, pins in MUTATIONS.values():
        for fn, args in pins:
            key = (fn.__name__, repr(args))
            if key not in seen:
                seen.add(key)
                fn(*args)
