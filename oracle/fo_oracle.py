"""FedOptima server-side oracle: a plain, slow, fp64 CPU statement of what the
server-side hot path computes.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this module:
only tests, ``__graft_entry__.smoke()`` and the CPU-baseline / reference arm
of ``bench.py`` may use it.  It shares no code with the CUDA library; both
consume only the seeded inputs of ``paper_2504_13850_gb300.workloads``.

What it follows (arxiv 2504.13850):
  * Task Scheduler ``put()`` (Algorithm 2) and ``get()`` with counter-based
    balancing (Algorithm 3, Sec. 3.3.2): models have priority, otherwise the
    device with the smallest consumption counter c_k is served and c_k += 1.
  * Activation flow control (Sec. 3.4.1): a global cap omega on the number of
    buffered batches, sum_k |Q_k| <= omega, and the "turn-on" signal sent to
    the device whose queue was enqueued to / dequeued from while the cap is
    not reached.  Server memory is model + omega batches (Eq. 3).
  * Server Compute Engine (Algorithm 4): one SGD training iteration on the
    server-side network per activation batch, and FedAsync aggregation of a
    local model with staleness cut-off D and weight alpha = 1/(t - t_k + 1).
  * Layer arithmetic is the textbook definition of each layer, in fp64;
    matrix products (numpy ``@``) are used as a library primitive.
  * The MobileNetV3 bottleneck pieces of the paper's testbed-B CNN
    (Table 4): depthwise convolution, hard swish, hard sigmoid and the
    squeeze-and-excite channel scaling (``dwconv_*``, ``hswish_*``,
    ``hsigmoid_*``, ``chmul_*``).  The derivatives at the kinks are a
    convention (the paper is silent): hard swish takes (2x + 3)/6 on the
    closed interval [-3, 3], 0 below and 1 above; hard sigmoid takes 1/6
    only strictly inside (-3, 3).  PyTorch 2.11 agrees on hard sigmoid but
    gives hard swish the open interval.
  * The Pre-processor's split point (Sec. 3.2, Eqs. 4-6): argmin over split
    points of the slowest device's max of training and transfer time
    (``split_point``; ties go to the smallest l).

Readings where the paper is silent (each one is listed in the design notes):
  * ties in argmin_k c_k go to the lowest k; only non-empty queues compete;
    a step with every queue empty returns EMPTY and changes nothing;
  * both the global cap omega and a per-device ring depth are enforced;
  * a device refused while its own queue is empty waits in a FIFO of
    blocked devices; each dequeue turns on the head of that FIFO;
  * free batch slots are handed out FIFO, starting 0..omega-1;
  * a device that (re)joins gets c_k = max(c_k, min over the other active
    devices' counters);
  * the server loss f_s is softmax cross-entropy averaged over the batch;
  * the server optimizer is SGD with momentum in the usual form
    v <- mu v + g, theta <- theta - lr v (v starts at 0);
  * ReLU'(0) = 0; a 2x2 max-pool sends its gradient to the first maximum in
    row-major window order;
  * the first server layer's input gradient is never formed: nothing is sent
    back to devices (gradient-free offloading, Sec. 3.2.2 / Sec. 3.3.1).

Two precisions.  With storage=None every value is fp64 (the definition).
With storage="bf16" the oracle keeps the same values a bf16 tensor-core
implementation stores, so that floating point takes every integer decision
(ReLU mask, max-pool argmax) in the kernel's precision: each op's output
and each activation gradient is rounded to bf16 (round to nearest even) when
stored, and the weights of every conv / linear layer except the logits layer
are rounded to bf16 before use; arithmetic in between stays fp64.
"""
from __future__ import annotations

from collections import deque

import numpy as np
from scipy.special import erf

OK, EMPTY, FULL, STALE = 0, 1, 2, 3
ERR_ARG = -1


def to_bf16(x):
    """Round to the nearest bfloat16 value (ties to even), returned as fp64.
    Rounds the fp64 value directly, without an intermediate fp32 step."""
    x = np.asarray(x, np.float64)
    m, e = np.frexp(x)                       # x = m * 2**e, 0.5 <= |m| < 1
    # bf16 keeps 8 significant bits: scale the mantissa to an integer grid
    return np.ldexp(np.round(np.ldexp(m, 8)), e - 8)


# ==========================================================================
# Task Scheduler: Algorithm 2 (put), Algorithm 3 (get), Sec. 3.4.1 (flow
# control)
# ==========================================================================

class TaskScheduler:
    """Activation side of the Task Scheduler.

    Q^act_k is a FIFO of batch-slot indices per device (Algorithm 2 puts the
    batch of device k = m.origin into Q^act_k).  ``get`` pops the head of the
    queue of the device with the smallest counter c_k (Algorithm 3) and
    increments c_k.  The model queue Q^model is served by the caller before
    each ``get`` (models have priority in Algorithm 3).
    """

    def __init__(self, K, omega, depth, policy="counter"):
        assert policy in ("counter", "fifo")
        self.K, self.omega, self.depth, self.policy = K, omega, depth, policy
        self.q = [deque() for _ in range(K)]
        self.c = [0] * K                     # batches consumed per device
        self.on = [True] * K                 # Sender Status of each device
        self.active = [True] * K
        self.free = deque(range(omega))      # free batch slots
        self.blocked = deque()               # refused with an empty queue
        self.arrivals = deque()              # device ids in arrival order (FIFO policy)

    def queued(self):
        return sum(len(q) for q in self.q)

    def put(self, k):
        """Algorithm 2, activation branch, with the server-side flow control of
        Sec. 3.4.1.  Returns (status, slot)."""
        if not (0 <= k < self.K) or not self.active[k]:
            return ERR_ARG, -1
        total = self.queued()
        if total >= self.omega or len(self.q[k]) >= self.depth:
            self.on[k] = False
            if not self.q[k] and k not in self.blocked:
                self.blocked.append(k)
            return FULL, -1
        slot = self.free.popleft()
        self.q[k].append(slot)
        if self.policy == "fifo":
            self.arrivals.append(k)
        if k in self.blocked:
            self.blocked.remove(k)
        # Enqueued to Q_k: turn device k on iff the cap is not reached.
        self.on[k] = (total + 1 < self.omega) and (len(self.q[k]) < self.depth)
        return OK, slot

    def get(self):
        """Algorithm 3, activation branch.  Returns (status, k, slot)."""
        if self.policy == "counter":
            cand = [k for k in range(self.K) if self.q[k]]
            if not cand:
                return EMPTY, -1, -1
            k = min(cand, key=lambda j: (self.c[j], j))      # argmin_k c_k
        else:
            if not self.arrivals:
                return EMPTY, -1, -1
            k = self.arrivals.popleft()
        slot = self.q[k].popleft()
        self.c[k] += 1
        self.free.append(slot)
        # Dequeued from Q_k: the cap is no longer reached, turn k on; one
        # device blocked with an empty queue is turned on as well.
        self.on[k] = True
        if self.blocked:
            self.on[self.blocked.popleft()] = True
        return OK, k, slot

    def set_active(self, k, active):
        if not (0 <= k < self.K):
            return ERR_ARG
        if active and not self.active[k]:
            others = [self.c[j] for j in range(self.K) if self.active[j] and j != k]
            if others:
                self.c[k] = max(self.c[k], min(others))
            self.active[k] = True
            self.on[k] = True
        elif not active and self.active[k]:
            self.active[k] = False
            self.on[k] = False
            if k in self.blocked:
                self.blocked.remove(k)
        return OK


# ==========================================================================
# FedAsync aggregation: Algorithm 4, aggregation branch
# ==========================================================================

class Aggregator:
    """Global device-side model version t and the staleness-weighted update
    theta_d <- alpha theta_dk + (1 - alpha) theta_d, alpha = 1/(t - t_k + 1),
    skipped when t - t_k > D.  theta_d and the auxiliary theta~_d are updated
    with the same alpha, so they are carried as one flat vector."""

    def __init__(self, K, max_delay):
        self.K, self.D, self.t = K, max_delay, 0

    def aggregate(self, theta_d, theta_dk, t_k):
        """Returns (status, new theta_d as fp64)."""
        if t_k < 0 or t_k > self.t:
            return ERR_ARG, theta_d
        if self.t - t_k > self.D:
            return STALE, theta_d
        alpha = 1.0 / (self.t - t_k + 1)
        g = np.asarray(theta_d, np.float64)
        l = np.asarray(theta_dk, np.float64)
        new = alpha * l + (1.0 - alpha) * g
        self.t += 1
        return OK, new

    @property
    def round(self):
        """Completed global rounds: a round ends after every K aggregations."""
        return self.t // self.K


# ==========================================================================
# Layers (fp64).  Image tensors are [B, H, W, C]; sequences [B, L, 1, d].
# ==========================================================================

def conv_fwd(x, w, b, stride, pad):
    """y[n,i,j,o] = b[o] + sum_{r,s,c} xpad[n, i*stride + r, j*stride + s, c] w[o,r,s,c]."""
    N, H, W, C = x.shape
    O, k, _, _ = w.shape
    Ho = (H + 2 * pad - k) // stride + 1
    Wo = (W + 2 * pad - k) // stride + 1
    xp = np.pad(x, ((0, 0), (pad, pad), (pad, pad), (0, 0)))
    y = np.zeros((N, Ho, Wo, O))
    for r in range(k):
        for s in range(k):
            win = xp[:, r:r + stride * (Ho - 1) + 1:stride, s:s + stride * (Wo - 1) + 1:stride, :]
            y += win @ w[:, r, s, :].T
    if b is not None:
        y += b
    return y


def conv_bwd(x, w, dy, stride, pad, need_dx):
    """Gradients of conv_fwd: (dx or None, dw, db)."""
    N, H, W, C = x.shape
    O, k, _, _ = w.shape
    _, Ho, Wo, _ = dy.shape
    xp = np.pad(x, ((0, 0), (pad, pad), (pad, pad), (0, 0)))
    dxp = np.zeros_like(xp) if need_dx else None
    dw = np.zeros_like(w)
    dy2 = dy.reshape(-1, O)
    for r in range(k):
        for s in range(k):
            sl = (slice(None), slice(r, r + stride * (Ho - 1) + 1, stride),
                  slice(s, s + stride * (Wo - 1) + 1, stride), slice(None))
            win = xp[sl]
            dw[:, r, s, :] = dy2.T @ win.reshape(-1, C)
            if need_dx:
                dxp[sl] += dy @ w[:, r, s, :]
    db = dy2.sum(axis=0)
    dx = dxp[:, pad:pad + H, pad:pad + W, :] if need_dx else None
    return dx, dw, db


def dwconv_fwd(x, w, b, stride, pad):
    """Depthwise convolution (one k x k filter per channel, as in the
    MobileNetV3 bottleneck): y[n,i,j,c] = b[c] +
    sum_{r,s} xpad[n, i*stride + r, j*stride + s, c] w[c,r,s]."""
    N, H, W, C = x.shape
    k = w.shape[1]
    Ho = (H + 2 * pad - k) // stride + 1
    Wo = (W + 2 * pad - k) // stride + 1
    xp = np.pad(x, ((0, 0), (pad, pad), (pad, pad), (0, 0)))
    y = np.zeros((N, Ho, Wo, C))
    for r in range(k):
        for s in range(k):
            y += xp[:, r:r + stride * (Ho - 1) + 1:stride, s:s + stride * (Wo - 1) + 1:stride, :] * w[:, r, s]
    if b is not None:
        y += b
    return y


def dwconv_bwd(x, w, dy, stride, pad, need_dx):
    """Gradients of dwconv_fwd: (dx or None, dw, db)."""
    N, H, W, C = x.shape
    k = w.shape[1]
    _, Ho, Wo, _ = dy.shape
    xp = np.pad(x, ((0, 0), (pad, pad), (pad, pad), (0, 0)))
    dxp = np.zeros_like(xp) if need_dx else None
    dw = np.zeros_like(w)
    for r in range(k):
        for s in range(k):
            sl = (slice(None), slice(r, r + stride * (Ho - 1) + 1, stride),
                  slice(s, s + stride * (Wo - 1) + 1, stride), slice(None))
            dw[:, r, s] = (dy * xp[sl]).sum(axis=(0, 1, 2))
            if need_dx:
                dxp[sl] += dy * w[:, r, s]
    db = dy.sum(axis=(0, 1, 2))
    dx = dxp[:, pad:pad + H, pad:pad + W, :] if need_dx else None
    return dx, dw, db


def hswish_fwd(x):
    """Hard swish x * relu6(x + 3) / 6."""
    return x * np.clip(x + 3.0, 0.0, 6.0) / 6.0


def hswish_bwd(x, dy):
    # derivative 0 below -3, (2x + 3) / 6 on [-3, 3], 1 above 3
    return dy * np.where(x < -3.0, 0.0, np.where(x > 3.0, 1.0, (2.0 * x + 3.0) / 6.0))


def hsigmoid_fwd(x):
    """Hard sigmoid relu6(x + 3) / 6."""
    return np.clip(x + 3.0, 0.0, 6.0) / 6.0


def hsigmoid_bwd(x, dy):
    # derivative 1/6 strictly inside (-3, 3), else 0
    return dy * np.where((x > -3.0) & (x < 3.0), 1.0 / 6.0, 0.0)


def chmul_fwd(x, s):
    """Channel scaling of the squeeze-and-excite block: y[n,h,w,c] = x[n,h,w,c] s[n,c]."""
    return x * s[:, None, None, :]


def chmul_bwd(x, s, dy):
    return dy * s[:, None, None, :], (dy * x).sum(axis=(1, 2))


def relu_fwd(x):
    return np.maximum(x, 0.0)


def relu_bwd(x, dy):
    return dy * (x > 0.0)                 # ReLU'(0) = 0


_POOL_ORDER = ((0, 0), (0, 1), (1, 0), (1, 1))   # row-major window order


def maxpool2_fwd(x):
    return np.maximum(np.maximum(x[:, 0::2, 0::2], x[:, 0::2, 1::2]),
                      np.maximum(x[:, 1::2, 0::2], x[:, 1::2, 1::2]))


def maxpool2_bwd(x, dy):
    """The gradient of each window goes to its first maximum (strict > scan)."""
    best = x[:, 0::2, 0::2].copy()
    arg = np.zeros(best.shape, np.int64)
    for t, (a, b) in enumerate(_POOL_ORDER[1:], start=1):
        cand = x[:, a::2, b::2]
        upd = cand > best
        best = np.where(upd, cand, best)
        arg = np.where(upd, t, arg)
    dx = np.zeros_like(x)
    for t, (a, b) in enumerate(_POOL_ORDER):
        dx[:, a::2, b::2] = np.where(arg == t, dy, 0.0)
    return dx


def affine_fwd(x, scale, shift):
    return x * scale + shift


def affine_bwd(x, scale, dy):
    c = x.shape[-1]
    return dy * scale, (dy * x).reshape(-1, c).sum(0), dy.reshape(-1, c).sum(0)


def linear_fwd(x, w, b):
    y = x @ w.T
    return y + b if b is not None else y


def linear_bwd(x, w, dy, need_dx):
    x2 = x.reshape(-1, x.shape[-1])
    dy2 = dy.reshape(-1, dy.shape[-1])
    dw = dy2.T @ x2
    db = dy2.sum(0)
    dx = dy @ w if need_dx else None
    return dx, dw, db


LN_EPS = 1e-5


def layernorm_fwd(x, gamma, beta):
    mu = x.mean(-1, keepdims=True)
    var = ((x - mu) ** 2).mean(-1, keepdims=True)      # biased variance
    rstd = 1.0 / np.sqrt(var + LN_EPS)
    xhat = (x - mu) * rstd
    return xhat * gamma + beta, (xhat, rstd)


def layernorm_bwd(cache, gamma, dy):
    xhat, rstd = cache
    c = xhat.shape[-1]
    dgamma = (dy * xhat).reshape(-1, c).sum(0)
    dbeta = dy.reshape(-1, c).sum(0)
    dxhat = dy * gamma
    dx = rstd * (dxhat - dxhat.mean(-1, keepdims=True)
                 - xhat * (dxhat * xhat).mean(-1, keepdims=True))
    return dx, dgamma, dbeta


def gelu_fwd(x):
    return x * 0.5 * (1.0 + erf(x / np.sqrt(2.0)))


def gelu_bwd(x, dy):
    cdf = 0.5 * (1.0 + erf(x / np.sqrt(2.0)))
    pdf = np.exp(-0.5 * x * x) / np.sqrt(2.0 * np.pi)
    return dy * (cdf + x * pdf)


def _split_heads(t, B, L, h, dh):
    return t.reshape(B, L, h, dh).transpose(0, 2, 1, 3)       # [B, h, L, dh]


def attention_fwd(qkv, lengths, d, heads):
    """Multi-head scaled dot-product attention over packed q|k|v [B, L, 1, 3d].
    Keys j >= lengths[b] are masked out.  Returns ([B, L, 1, d], cache)."""
    B, L = qkv.shape[0], qkv.shape[1]
    dh = d // heads
    t = qkv.reshape(B, L, 3 * d)
    q = _split_heads(t[..., :d], B, L, heads, dh)
    k = _split_heads(t[..., d:2 * d], B, L, heads, dh)
    v = _split_heads(t[..., 2 * d:], B, L, heads, dh)
    s = q @ k.transpose(0, 1, 3, 2) / np.sqrt(dh)
    valid = np.arange(L)[None, :] < np.asarray(lengths)[:, None]      # [B, L] keys
    s = np.where(valid[:, None, None, :], s, -np.inf)
    s = s - s.max(-1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(-1, keepdims=True)
    o = p @ v                                                      # [B, h, L, dh]
    out = o.transpose(0, 2, 1, 3).reshape(B, L, 1, d)
    return out, (q, k, v, p)


def attention_bwd(cache, dout, d, heads):
    q, k, v, p = cache
    B, h, L, dh = q.shape
    do = _split_heads(dout.reshape(B, L, d), B, L, h, dh)
    dv = p.transpose(0, 1, 3, 2) @ do
    dp = do @ v.transpose(0, 1, 3, 2)
    ds = p * (dp - (p * dp).sum(-1, keepdims=True))
    dq = ds @ k / np.sqrt(dh)
    dk = ds.transpose(0, 1, 3, 2) @ q / np.sqrt(dh)
    merge = lambda t: t.transpose(0, 2, 1, 3).reshape(B, L, d)
    return np.concatenate([merge(dq), merge(dk), merge(dv)], -1).reshape(B, L, 1, 3 * d)


def meanpool_fwd(x, lengths):
    """Mean over the valid tokens of each sequence: [B, L, 1, d] -> [B, d]."""
    B, L = x.shape[0], x.shape[1]
    y = np.zeros((B, x.shape[-1]))
    for b in range(B):
        y[b] = x[b, :lengths[b], 0, :].mean(0)
    return y


def meanpool_bwd(x, lengths, dy):
    dx = np.zeros_like(x)
    for b in range(x.shape[0]):
        dx[b, :lengths[b], 0, :] = dy[b] / lengths[b]
    return dx


def avgpool_fwd(x):
    return x.mean(axis=(1, 2))


def avgpool_bwd(x, dy):
    N, H, W, C = x.shape
    return np.broadcast_to(dy[:, None, None, :] / (H * W), x.shape).copy()


def softmax_ce(z, labels):
    """f_s: softmax cross-entropy, mean over the batch (natural log).
    Returns (loss, dL/dz)."""
    B, C = z.shape
    m = z.max(-1, keepdims=True)
    e = np.exp(z - m)
    se = e.sum(-1, keepdims=True)
    lse = m[:, 0] + np.log(se[:, 0])
    loss = float(np.mean(lse - z[np.arange(B), labels]))
    dz = e / se
    dz[np.arange(B), labels] -= 1.0
    return loss, dz / B


# ==========================================================================
# Server-side network: Algorithm 4, training branch
# ==========================================================================

def param_shapes(ops):
    """Parameter tensors in flat order: conv W[cout][k][k][cin] (+ b), linear
    W[cout][cin] (+ b), affine scale, shift, layernorm gamma, beta."""
    out = []
    for i, op in enumerate(ops):
        kd = op["kind"]
        if kd == "conv":
            out.append((i, "W", (op["cout"], op["k"], op["k"], op["cin"])))
            if op["bias"]:
                out.append((i, "b", (op["cout"],)))
        elif kd == "linear":
            out.append((i, "W", (op["cout"], op["cin"])))
            if op["bias"]:
                out.append((i, "b", (op["cout"],)))
        elif kd == "affine":
            out.append((i, "scale", (op["c"],)))
            out.append((i, "shift", (op["c"],)))
        elif kd == "layernorm":
            out.append((i, "gamma", (op["c"],)))
            out.append((i, "beta", (op["c"],)))
        elif kd == "dwconv":
            out.append((i, "W", (op["c"], op["k"], op["k"])))
            if op["bias"]:
                out.append((i, "b", (op["c"],)))
    return out


def unflatten(ops, flat):
    params, off = {}, 0
    for i, name, shape in param_shapes(ops):
        n = int(np.prod(shape))
        params[(i, name)] = np.asarray(flat[off:off + n], np.float64).reshape(shape)
        off += n
    assert off == len(flat), (off, len(flat))
    return params


def flatten(ops, grads):
    return np.concatenate([grads[(i, name)].ravel() for i, name, _ in param_shapes(ops)])


def _weights(ops, params, i, storage):
    w = params.get((i, "W"))
    if storage == "bf16" and i < len(ops) - 1:
        w = to_bf16(w)
    return w


def forward(ops, params, x, lengths, storage=None):
    """Forward pass of M_s.  Returns the list of tensors (tensor 0 = x) and
    per-op caches."""
    T = [np.asarray(x, np.float64)]
    caches = [None] * len(ops)
    for i, op in enumerate(ops):
        kd, a = op["kind"], T[op["in0"]]
        P = lambda n: _weights(ops, params, i, storage) if n == "W" else params.get((i, n))
        if kd == "conv":
            y = conv_fwd(a, P("W"), P("b"), op["stride"], op["k"] // 2)
        elif kd == "affine":
            y = affine_fwd(a, P("scale"), P("shift"))
        elif kd == "relu":
            y = relu_fwd(a)
        elif kd == "maxpool2":
            y = maxpool2_fwd(a)
        elif kd == "add":
            y = a + T[op["in1"]]
        elif kd == "avgpool":
            y = avgpool_fwd(a)
        elif kd == "flatten":
            y = a.reshape(a.shape[0], -1)
        elif kd == "linear":
            y = linear_fwd(a, P("W"), P("b"))
        elif kd == "layernorm":
            y, caches[i] = layernorm_fwd(a, P("gamma"), P("beta"))
        elif kd == "gelu":
            y = gelu_fwd(a)
        elif kd == "attention":
            y, caches[i] = attention_fwd(a, lengths, op["c"], op["heads"])
        elif kd == "meanpool":
            y = meanpool_fwd(a, lengths)
        elif kd == "dwconv":
            y = dwconv_fwd(a, P("W"), P("b"), op["stride"], op["k"] // 2)
        elif kd == "hswish":
            y = hswish_fwd(a)
        elif kd == "hsigmoid":
            y = hsigmoid_fwd(a)
        elif kd == "chmul":
            y = chmul_fwd(a, T[op["in1"]])
        else:
            raise ValueError(kd)
        if storage == "bf16" and i < len(ops) - 1:
            y = to_bf16(y)
        T.append(y)
    return T, caches


def backward(ops, params, T, caches, dlogits, lengths, storage=None):
    """Backward pass of M_s.  The input tensor (tensor 0) receives no
    gradient: the server never returns gradients to devices.  Contributions
    to a tensor's gradient are added in reverse op order."""
    G = {len(ops): dlogits}
    grads = {}
    rnd = to_bf16 if storage == "bf16" else (lambda v: v)

    def acc(tid, g):
        if tid == 0 or g is None:
            return
        G[tid] = rnd(G[tid] + g) if tid in G else rnd(g)

    for i in range(len(ops) - 1, -1, -1):
        op = ops[i]
        kd, a = op["kind"], T[op["in0"]]
        dy = G.pop(i + 1, None)
        if dy is None:
            dy = np.zeros_like(T[i + 1])
        need = op["in0"] != 0
        P = lambda n: _weights(ops, params, i, storage) if n == "W" else params.get((i, n))
        if kd == "conv":
            dx, dw, db = conv_bwd(a, P("W"), dy, op["stride"], op["k"] // 2, need)
            grads[(i, "W")] = dw
            if op["bias"]:
                grads[(i, "b")] = db
            acc(op["in0"], dx)
        elif kd == "affine":
            dx, ds, dsh = affine_bwd(a, P("scale"), dy)
            grads[(i, "scale")], grads[(i, "shift")] = ds, dsh
            acc(op["in0"], dx)
        elif kd == "relu":
            acc(op["in0"], relu_bwd(a, dy))
        elif kd == "maxpool2":
            acc(op["in0"], maxpool2_bwd(a, dy))
        elif kd == "add":
            acc(op["in0"], dy)
            acc(op["in1"], dy)
        elif kd == "avgpool":
            acc(op["in0"], avgpool_bwd(a, dy))
        elif kd == "flatten":
            acc(op["in0"], dy.reshape(a.shape))
        elif kd == "linear":
            dx, dw, db = linear_bwd(a, P("W"), dy, need)
            grads[(i, "W")] = dw
            if op["bias"]:
                grads[(i, "b")] = db
            acc(op["in0"], dx)
        elif kd == "layernorm":
            dx, dg, dbt = layernorm_bwd(caches[i], P("gamma"), dy)
            grads[(i, "gamma")], grads[(i, "beta")] = dg, dbt
            acc(op["in0"], dx)
        elif kd == "gelu":
            acc(op["in0"], gelu_bwd(a, dy))
        elif kd == "attention":
            acc(op["in0"], attention_bwd(caches[i], dy, op["c"], op["heads"]))
        elif kd == "meanpool":
            acc(op["in0"], meanpool_bwd(a, lengths, dy))
        elif kd == "dwconv":
            dx, dw, db = dwconv_bwd(a, P("W"), dy, op["stride"], op["k"] // 2, need)
            grads[(i, "W")] = dw
            if op["bias"]:
                grads[(i, "b")] = db
            acc(op["in0"], dx)
        elif kd == "hswish":
            acc(op["in0"], hswish_bwd(a, dy))
        elif kd == "hsigmoid":
            acc(op["in0"], hsigmoid_bwd(a, dy))
        elif kd == "chmul":
            dx, ds = chmul_bwd(a, T[op["in1"]], dy)
            acc(op["in0"], dx)
            acc(op["in1"], ds)
        else:
            raise ValueError(kd)
    return grads


def loss_and_grad(ops, theta, x, labels, lengths=None, storage=None):
    """f_s(theta_s; xi) and its gradient (flat fp64)."""
    params = unflatten(ops, theta)
    T, caches = forward(ops, params, x, lengths, storage)
    loss, dz = softmax_ce(T[-1], np.asarray(labels))
    grads = backward(ops, params, T, caches, dz, lengths, storage)
    return loss, flatten(ops, grads)


def sgd_momentum(theta, v, g, lr, mu):
    """theta_s <- theta_s - gamma_s * v with v <- mu v + g."""
    v = mu * v + g
    return theta - lr * v, v


def server_step(ops, theta, v, x, labels, lengths, lr, mu, storage=None):
    """One training iteration of Algorithm 4 (forward, loss, backward,
    update).  Returns (loss, theta, v, g)."""
    loss, g = loss_and_grad(ops, theta, x, labels, lengths, storage)
    theta, v = sgd_momentum(np.asarray(theta, np.float64), np.asarray(v, np.float64), g, lr, mu)
    return loss, theta, v, g


# ==========================================================================
# Event replay: the server's view of a run
# ==========================================================================

class Server:
    """The server state the paper's algorithms act on: scheduler, one-copy
    server model (theta_s, momentum), batch slots and the aggregator."""

    def __init__(self, ops, K, omega, depth, theta0, lr, mu, max_delay=2**31 - 1,
                 policy="counter", storage=None):
        self.ops = ops
        self.storage = storage
        self.sched = TaskScheduler(K, omega, depth, policy)
        self.agg = Aggregator(K, max_delay)
        self.theta = np.asarray(theta0, np.float64).copy()
        self.v = np.zeros_like(self.theta)
        self.lr, self.mu = lr, mu
        self.slots = {}
        self.losses = []

    def enqueue(self, k, acts, labels, lengths=None):
        st, slot = self.sched.put(k)
        if st == OK:
            # uploads are fp32 / bf16 values: kept as given, widened to fp64 at use
            self.slots[slot] = (np.array(acts, copy=True), np.asarray(labels),
                                None if lengths is None else np.asarray(lengths))
        return st, slot

    def step(self):
        st, k, slot = self.sched.get()
        if st != OK:
            return st, -1, -1
        x, y, ln = self.slots.pop(slot)
        loss, self.theta, self.v, _ = server_step(self.ops, self.theta, self.v, x, y, ln,
                                                  self.lr, self.mu, self.storage)
        self.losses.append(loss)
        return OK, k, slot

    def aggregate(self, theta_d, theta_dk, t_k):
        return self.agg.aggregate(theta_d, theta_dk, t_k)


# ---------------------------------------------------------------------------
# Pre-processor (Sec. 3.2, "Splitting the DNN", Eqs. 4-6)
# ---------------------------------------------------------------------------
def split_point(O, S, b, o, allowed=None):
    """Split point l (1-based: M_d = layers 1..l) minimising, over the
    candidate points, the slowest device's max of its training time
    t_train_k(l) = sum_{i<=l} O_i / o_k (Eq. 4) and its activation transfer
    time t_transfer_k(l) = S_l / b_k (Eq. 5); Eq. 6 takes the argmin over l
    of the max over devices.  Candidates: every l, or those with
    allowed[l-1] true.  Ties: smallest l (the paper is silent).
    Returns (l, cost in seconds)."""
    L, K = len(O), len(b)
    best_l, best_cost = None, None
    for l in range(1, L + 1):
        if allowed is not None and not allowed[l - 1]:
            continue
        worst = 0.0
        for k in range(K):
            t_train = sum(float(O[i]) for i in range(l)) / float(o[k])
            t_transfer = float(S[l - 1]) / float(b[k])
            worst = max(worst, t_train, t_transfer)
        if best_cost is None or worst < best_cost:
            best_l, best_cost = l, worst
    return best_l, best_cost
