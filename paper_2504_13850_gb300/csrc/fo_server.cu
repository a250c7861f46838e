// FedOptima server: C-ABI entry points, HBM activation slab, one-copy
// server model and the step plan (forward, loss, backward, optimizer).
//
// Memory (Eq. 3 of the paper): one copy of theta_s (+ momentum, gradient,
// bf16 shadow) and `omega` activation batch slots, independent of the
// number of devices K.  Q^act_k are rings of slot indices on the host
// (fo_sched.hpp); a slot's bytes live in the slab until the step that
// consumes it has finished reading them (CUDA events order the reuse).
#include "fo_server_impl.h"

#include <memory>
#include "fo_tc.h"

#include <cstring>
#include <functional>
#include <map>
#include <new>
#include <string>
#include <vector>

namespace {

thread_local std::string g_err;

int set_err(int code, const std::string& msg) {
  g_err = msg;
  return code;
}

#define FO_CUDA(call)                                                                   \
  do {                                                                                  \
    cudaError_t e_ = (call);                                                            \
    if (e_ != cudaSuccess)                                                              \
      return set_err(FO_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

}  // namespace

namespace fo {
// Records `msg` as the calling thread's fo_last_error() and returns `code`.
int report_error(int code, const std::string& msg) { return set_err(code, msg); }
}  // namespace fo

namespace {

int64_t pad64(int64_t n) { return (n + 63) / 64 * 64; }

// Weight tensors of at least this many parameters get their own update as
// soon as their gradient is final; smaller ones (where a launch costs more
// than the traffic it moves) are left to the step's final update.
constexpr int64_t kEarlyUpdateMin = 128 * 1024;
// Early updates are batched: consecutive weight tensors share one launch once
// they add up to this many parameters (or the segment table is full).
constexpr int64_t kEarlyGroupMin = 2 * 1024 * 1024;

// Shape inference and parameter layout.  Returns FO_OK or an error.
int infer(fo_server* s) {
  const fo_server_cfg& c = s->cfg;
  int nops = int(s->ops.size());
  s->T.assign(nops + 1, Tensor());
  Tensor& t0 = s->T[0];
  t0.N = c.batch;
  t0.H = c.in_h;
  t0.W = c.in_w;
  t0.C = c.in_c;
  t0.dt = s->dt;
  t0.root = 0;
  s->op_segs.assign(nops, {});
  int64_t off = 0, flat = 0;
  auto add_seg = [&](int i, int64_t n) {
    s->op_segs[i].push_back(int(s->segs.size()));
    s->segs.push_back({i, off, flat, n});
    off += pad64(n);
    flat += n;
  };
  for (int i = 0; i < nops; ++i) {
    const fo_op& op = s->ops[i];
    if (op.in0 < 0 || op.in0 > i) return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": bad in0");
    const Tensor& a = s->T[op.in0];
    Tensor o = a;
    o.act = o.grad = nullptr;
    o.root = i + 1;
    o.consumers = 0;
    o.dt = s->dt;
    switch (op.kind) {
      case FO_OP_CONV: {
        if (a.C != op.cin || (op.k != 1 && op.k != 3) || (op.stride != 1 && op.stride != 2) || op.cout <= 0)
          return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": bad conv");
        int pad = op.k / 2;
        o.H = (a.H + 2 * pad - op.k) / op.stride + 1;
        o.W = (a.W + 2 * pad - op.k) / op.stride + 1;
        o.C = op.cout;
        add_seg(i, int64_t(op.cout) * op.k * op.k * op.cin);
        if (op.bias) add_seg(i, op.cout);
        break;
      }
      case FO_OP_AFFINE:
        if (a.C != op.cin) return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": affine channels");
        add_seg(i, op.cin);
        add_seg(i, op.cin);
        break;
      case FO_OP_RELU:
      case FO_OP_GELU:
        break;
      case FO_OP_MAXPOOL2:
        if (a.H % 2 || a.W % 2) return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": maxpool odd size");
        o.H = a.H / 2;
        o.W = a.W / 2;
        break;
      case FO_OP_ADD: {
        if (op.in1 < 0 || op.in1 > i) return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": bad in1");
        const Tensor& b = s->T[op.in1];
        if (b.N != a.N || b.H != a.H || b.W != a.W || b.C != a.C)
          return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": add shapes differ");
        break;
      }
      case FO_OP_AVGPOOL:
        o.H = o.W = 1;
        break;
      case FO_OP_FLATTEN:
        o.C = a.H * a.W * a.C;
        o.H = o.W = 1;
        o.root = s->T[op.in0].root;
        break;
      case FO_OP_LINEAR:
        if (a.C != op.cin || op.cout <= 0) return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": linear cin");
        o.C = op.cout;
        add_seg(i, int64_t(op.cout) * op.cin);
        if (op.bias) add_seg(i, op.cout);
        break;
      case FO_OP_LAYERNORM:
        if (a.C != op.cin || a.C % 32) return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": layernorm channels");
        add_seg(i, op.cin);
        add_seg(i, op.cin);
        break;
      case FO_OP_ATTENTION:
        if (a.C != 3 * op.cin || op.heads <= 0 || op.cin % op.heads || op.cin / op.heads > 64 ||
            a.H > 128 || a.W != 1 || !c.seq)
          return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": attention shape");
        o.C = op.cin;
        break;
      case FO_OP_MEANPOOL:
        if (a.W != 1 || !c.seq) return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": meanpool shape");
        o.H = 1;
        break;
      case FO_OP_DWCONV: {
        if (a.C != op.cin || op.k < 1 || op.k > 7 || op.k % 2 == 0 || (op.stride != 1 && op.stride != 2))
          return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": bad depthwise conv");
        int pad = op.k / 2;
        o.H = (a.H + 2 * pad - op.k) / op.stride + 1;
        o.W = (a.W + 2 * pad - op.k) / op.stride + 1;
        add_seg(i, int64_t(op.cin) * op.k * op.k);
        if (op.bias) add_seg(i, op.cin);
        break;
      }
      case FO_OP_HSWISH:
      case FO_OP_HSIGMOID:
        break;
      case FO_OP_CHMUL: {
        if (op.in1 < 0 || op.in1 > i) return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": bad in1");
        const Tensor& b = s->T[op.in1];
        if (b.N != a.N || b.H != 1 || b.W != 1 || b.C != a.C)
          return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": channel scale must be [B, 1, 1, C]");
        break;
      }
      default:
        return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": unknown kind");
    }
    if (int64_t(o.H) * o.W * o.C > INT32_MAX)
      return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": more than 2^31 - 1 elements per sample");
    s->T[i + 1] = o;
    s->T[op.in0].consumers++;
    if (op.kind == FO_OP_ADD || op.kind == FO_OP_CHMUL) s->T[op.in1].consumers++;
  }
  const fo_op& last = s->ops.back();
  const Tensor& lt = s->T.back();
  if (last.kind != FO_OP_LINEAR || lt.rows() != c.batch || lt.C != c.num_classes)
    return set_err(FO_ERR_ARG, "the last op must be a linear layer producing [batch, num_classes]");
  s->T.back().dt = fo::kF32;  // logits
  s->n_params = flat;
  s->n_padded = off;
  return FO_OK;
}

float* P(fo_server* s, int op, int which) { return s->theta + s->segs[s->op_segs[op][which]].off; }
float* G(fo_server* s, int op, int which) { return s->grad + s->segs[s->op_segs[op][which]].off; }
const fo::bf16* SH(fo_server* s, int op, int which) { return s->shadow + s->segs[s->op_segs[op][which]].off; }

fo::ConvShape conv_shape(const fo_server* s, int i) {
  const fo_op& op = s->ops[i];
  const Tensor& a = s->T[op.in0];
  const Tensor& o = s->T[i + 1];
  if (op.kind == FO_OP_LINEAR)
    return {int(a.rows()), 1, 1, op.cin, op.cout, 1, 1, 0, 1, 1};
  return {a.N, a.H, a.W, op.cin, op.cout, op.k, op.stride, op.k / 2, o.H, o.W};
}

fo::DwShape dw_shape(const fo_server* s, int i) {
  const fo_op& op = s->ops[i];
  const Tensor& a = s->T[op.in0];
  const Tensor& o = s->T[i + 1];
  return {a.N, a.H, a.W, op.cin, op.k, op.stride, op.k / 2, o.H, o.W};
}

// Which kernels absorb which neighbouring work (decided once per network).
struct Fusion {
  std::vector<int> fwd_relu;   // producer op -> the relu op it applies, or -1
  std::vector<char> skip_fwd;  // relu op whose forward is done by its producer
  std::vector<int> bwd_mask;   // consumer op -> relu op whose mask it applies to its dx, or -1
  std::vector<char> skip_bwd;  // relu op whose backward is done by its consumer
  std::vector<int> hswish_of;  // affine op -> the hard swish op it applies (both passes), or -1
  std::vector<int> hswish_by;  // hard swish op -> the affine op that applies it, or -1
  std::vector<int> add_relu;   // residual add op -> the relu after it, whose backward the add's applies, or -1
  std::vector<int> relu_into_add;  // that relu op -> the add op, or -1
  // Residual add whose branch ends in a plain tensor-core GEMM: the GEMM's
  // epilogue writes branch + residual straight into the add's output, the
  // branch's gradient is the add's output gradient itself (one buffer), and
  // the residual's gradient joins its next contribution as an addend.
  std::vector<int> add_into;   // producer op -> the add op whose output it writes, or -1
  std::vector<int> add_other;  // that add op -> its residual operand tensor
  std::vector<int> branch_of;  // that add op -> its branch tensor, or -1
  // A linear layer whose output feeds only a GELU: its epilogue may store
  // the GELU too (the plan decides; the GELU op runs alone otherwise).
  std::vector<int> gelu_of;    // producer op -> the GELU op, or -1
  bool head = false;           // last linear + loss handled by the head kernels
};

bool dx_takes_mask(const fo_server* s, int j) {
  const fo_op& op = s->ops[j];
  return op.kind == FO_OP_CONV || op.kind == FO_OP_LINEAR || op.kind == FO_OP_MAXPOOL2;
}

Fusion analyse(const fo_server* s) {
  const int nops = int(s->ops.size());
  Fusion f;
  f.fwd_relu.assign(nops, -1);
  f.skip_fwd.assign(nops, 0);
  f.bwd_mask.assign(nops, -1);
  f.skip_bwd.assign(nops, 0);
  f.gelu_of.assign(nops, -1);
  f.hswish_of.assign(nops, -1);
  f.hswish_by.assign(nops, -1);
  f.add_relu.assign(nops, -1);
  f.relu_into_add.assign(nops, -1);
  f.add_into.assign(nops, -1);
  f.add_other.assign(nops, -1);
  f.branch_of.assign(nops, -1);
  std::vector<int> sole(nops + 1, -1);  // the only consumer op of a tensor
  for (int j = 0; j < nops; ++j) {
    const fo_op& op = s->ops[j];
    if (s->T[op.in0].consumers == 1) sole[op.in0] = j;
    if (op.kind == FO_OP_ADD && s->T[op.in1].consumers == 1) sole[op.in1] = j;
  }
  const fo_op& last = s->ops.back();
  f.head = last.kind == FO_OP_LINEAR && s->cfg.num_classes <= 1024;
  for (int r = 0; r < nops; ++r) {
    const fo_op& op = s->ops[r];
    if (op.kind != FO_OP_RELU || s->T[op.in0].is_input()) continue;
    const int p = op.in0 - 1;  // producer op of the relu input
    const int pk = s->ops[p].kind;
    if (sole[op.in0] == r && (pk == FO_OP_CONV || pk == FO_OP_LINEAR || pk == FO_OP_AFFINE || pk == FO_OP_ADD) &&
        !(f.head && p == nops - 1)) {
      f.fwd_relu[p] = r;
      f.skip_fwd[r] = 1;
    }
    const int j = sole[r + 1];
    if (j >= 0 && s->ops[j].in0 == r + 1 && (dx_takes_mask(s, j) || (f.head && j == nops - 1))) {
      f.bwd_mask[j] = r;
      f.skip_bwd[r] = 1;
    }
  }
  // A relu whose input is a residual add's output (and that add's only
  // consumer), not already applied by its own consumer: the add's backward
  // masks the relu output's gradient on the fly and writes both inputs.
  for (int r = 0; r < nops; ++r) {
    const fo_op& op = s->ops[r];
    if (op.kind != FO_OP_RELU || s->T[op.in0].is_input() || f.skip_bwd[r]) continue;
    const int p = op.in0 - 1;
    if (s->ops[p].kind == FO_OP_ADD && sole[op.in0] == r) {
      f.add_relu[p] = r;
      f.relu_into_add[r] = p;
    }
  }
  // A batch-norm affine whose only consumer is a hard swish (the MobileNetV3
  // bottleneck) applies it in both passes, on the vectorised bf16 path.
  for (int h = 0; h < nops; ++h) {
    const fo_op& op = s->ops[h];
    if (op.kind != FO_OP_HSWISH || s->T[op.in0].is_input()) continue;
    const int p = op.in0 - 1;
    const Tensor& t = s->T[op.in0];
    if (s->ops[p].kind == FO_OP_AFFINE && sole[op.in0] == h && f.fwd_relu[p] < 0 && fo::vec8_ok(s->dt, t.numel()) &&
        t.C % 8 == 0) {
      f.hswish_of[p] = h;
      f.hswish_by[h] = p;
      f.skip_fwd[h] = 1;
    }
  }
  const int L = nops - 1;
  auto plain = [&](int j) { return fo::tc_plain_ok(s->tc, s, j) && !(f.head && j == L); };
  for (int a = 0; a < nops; ++a) {
    const fo_op& op = s->ops[a];
    if (op.kind != FO_OP_ADD || f.fwd_relu[a] >= 0 || f.add_relu[a] >= 0) continue;
    for (int t : {op.in1, op.in0}) {
      const int other = t == op.in1 ? op.in0 : op.in1;
      if (s->T[t].is_input() || s->T[t].root != t || s->T[t].root == s->T[other].root || sole[t] != a) continue;
      const int p = t - 1;
      if (!plain(p) || f.fwd_relu[p] >= 0) continue;
      f.add_into[p] = a;
      f.add_other[a] = other;
      f.branch_of[a] = t;
      f.skip_fwd[a] = 1;
      break;
    }
  }
  for (int g = 0; g < nops && !getenv("FO_NO_GELU_EPILOGUE"); ++g) {
    const fo_op& op = s->ops[g];
    if (op.kind != FO_OP_GELU || s->T[op.in0].is_input()) continue;
    const int p = op.in0 - 1;
    if (s->ops[p].kind == FO_OP_LINEAR && sole[op.in0] == g && plain(p) && f.fwd_relu[p] < 0 && f.add_into[p] < 0)
      f.gelu_of[p] = g;
  }
  return f;
}

// Build the list of launches of one server step.  Every entry records how
// many kernels it launches and its algorithmic FLOPs / HBM bytes (the
// minimum a kernel of that job must move), for the per-kernel roofline.
// A ReLU is applied by the kernel producing its input (forward) and by the
// kernel producing its output gradient (backward): the mask y > 0 of the
// ReLU output equals x > 0 of its input.
int build_plan(fo_server* s) {
  const int nops = int(s->ops.size());
  const int dt = s->dt;
  const double esz = dt == fo::kF32 ? 4.0 : 2.0;
  auto& plan = s->plan;
  plan.clear();
  for (fo::AttnTcPlan* a : s->attn_tc) fo::attention_tc_destroy(a);
  s->attn_tc.assign(nops, nullptr);
  const Fusion fu = analyse(s);
  for (int i = 0; i < nops; ++i)   // a fused residual's branch shares the add's output gradient
    if (fu.branch_of[i] >= 0) s->T[fu.branch_of[i]].grad = s->T[i + 1].grad;
  auto act = [s](int tid) -> const void* { return s->T[tid].is_input() ? s->cur_in : s->T[tid].act; };
  auto add = [&plan](const char* name, int kernels, double flops, double bytes,
                     std::function<void(cudaStream_t)> fn, int lane = 0) {
    plan.push_back({name, std::move(fn), kernels, flops, bytes, lane});
  };
  auto tbytes = [s](int tid) { return double(s->T[tid].bytes()); };
  auto add_tc = [&](fo::TcGemm* g, int lane = 0) {
    fo::tc_set_lane(g, lane);
    add(fo::tc_name(g), 1, fo::tc_flops(g), 0.0, [=](cudaStream_t st) { fo::tc_run(g, nullptr, st); }, lane);
  };
  const int L = nops - 1;  // the logits layer

  // Max-pools computed by the epilogue of the conv / linear in front of them
  // (through its ReLU): per pool op, the window codes that epilogue stores,
  // or null.
  std::vector<uint8_t*> pool_codes(nops, nullptr);
  std::vector<char> gelu_done(nops, 0);   // GELU ops stored by the producing GEMM's epilogue

  // ---------------- forward
  for (int i = 0; i < nops; ++i) {
    const fo_op op = s->ops[i];
    if (fu.skip_fwd[i] || pool_codes[i]) continue;
    const int a = op.in0;
    // output buffer: a fused relu writes the relu's output tensor, a fused
    // residual add the add's output
    const int o = fu.fwd_relu[i] >= 0 ? fu.fwd_relu[i] + 1 : (fu.add_into[i] >= 0 ? fu.add_into[i] + 1 : i + 1);
    const bool relu = fu.fwd_relu[i] >= 0;
    const Tensor& ta = s->T[a];
    const Tensor& to = s->T[i + 1];
    if (fu.head && i == L) {
      // logits, loss, dz and (when the input needs one) the input gradient:
      // the classifier is the first op of the backward pass, so that
      // gradient is its destination's first contribution
      const int B = s->cfg.batch, K = op.cin, C = op.cout;
      const int mr = fu.bwd_mask[i];
      const int da = mr >= 0 ? s->ops[mr].in0 : a;
      const void* mask = mr >= 0 ? s->T[mr + 1].act : nullptr;
      const bool dx = !s->T[a].is_input();
      add("head_fwd_ce", 1, 2.0 * B * K * C * (dx ? 2.0 : 1.0), tbytes(a) * (dx ? 3.0 : 1.0), [=](cudaStream_t st) {
        fo::head_forward_loss(act(a), s->T[a].dt, P(s, i, 0), op.bias ? P(s, i, 1) : nullptr, s->cur_labels, B,
                              K, C, (float*)s->T[i + 1].act, (float*)s->T[i + 1].grad, s->row_loss, st, mask,
                              dx ? s->T[da].grad : nullptr, false);
      });
      continue;
    }
    switch (op.kind) {
      case FO_OP_CONV:
      case FO_OP_LINEAR: {
        fo::ConvShape cs = conv_shape(s, i);
        const bool bias = op.bias != 0;
        const double fl = 2.0 * double(to.rows()) * op.cout * double(op.kind == FO_OP_CONV ? op.k * op.k : 1) * op.cin;
        fo::TcEpilogue ex;
        const bool fused = fu.add_into[i] >= 0;
        if (fused) {
          const int r = fu.add_other[fu.add_into[i]];
          if (s->T[r].is_input()) ex.addend_is_input = true;
          else ex.addend = s->T[r].act;
        }
        fo::TcGemm* tg = nullptr;
        // ReLU then a 2x2 max-pool that alone reads the ReLU output and applies
        // its mask in the backward pass: the pool goes into this epilogue
        const int pr = fu.fwd_relu[i];
        int pq = -1;
        if (pr >= 0 && !fused && dt == fo::kBF16 && s->T[pr + 1].consumers == 1 && !getenv("FO_NO_POOL_EPILOGUE"))
          for (int q = pr + 1; q < nops; ++q)
            if (s->ops[q].in0 == pr + 1) {
              if (s->ops[q].kind == FO_OP_MAXPOOL2 && fu.bwd_mask[q] == pr) pq = q;
              break;
            }
        if (pq >= 0) {
          const Tensor& tp = s->T[pq + 1];
          uint8_t* codes = (uint8_t*)s->alloc(size_t(tp.numel()));
          if (!codes) return set_err(FO_ERR_OOM, "max-pool window codes");
          ex.pool_out = tp.act;
          ex.pool_code = codes;
          tg = fo::tc_plan_forward(s->tc, s, i, s->T[o].act, relu, &ex);
          if (tg) pool_codes[pq] = codes;
          ex.pool_out = nullptr;
          ex.pool_code = nullptr;
        }
        if (!tg && fu.gelu_of[i] >= 0) {
          ex.gelu_out = s->T[fu.gelu_of[i] + 1].act;
          tg = fo::tc_plan_forward(s->tc, s, i, s->T[o].act, relu, &ex);
          if (tg) gelu_done[fu.gelu_of[i]] = 1;
          ex.gelu_out = nullptr;
        }
        if (!tg) tg = fo::tc_plan_forward(s->tc, s, i, s->T[o].act, relu, fused ? &ex : nullptr);
        if (fused && !tg) return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": fused epilogue not planned");
        if (tg) {
          add_tc(tg);
        } else {
          // Hidden layers of the bf16 path multiply bf16 weights (the shadow);
          // the fp32 path and the fp32 logits layer use the fp32 master.
          const int dto = to.dt;
          const bool wbf = dto == fo::kBF16;
          add(op.kind == FO_OP_CONV ? "conv_fwd_simt" : "linear_fwd_simt", 1, fl, 0.0, [=](cudaStream_t st) {
            const void* w = wbf ? (const void*)SH(s, i, 0) : (const void*)P(s, i, 0);
            fo::conv_fwd_simt(cs, act(a), ta.dt, w, wbf ? fo::kBF16 : fo::kF32, bias ? P(s, i, 1) : nullptr,
                              s->T[o].act, dto, relu, st);
          });
        }
        break;
      }
      case FO_OP_AFFINE:
        if (fu.hswish_of[i] >= 0) {
          const int h = fu.hswish_of[i] + 1;   // the hard swish's output tensor
          add("affine_hswish_fwd", 1, 0.0, 3 * tbytes(a), [=](cudaStream_t st) {
            fo::affine_hswish_fwd_x8(act(a), P(s, i, 0), P(s, i, 1), s->T[o].act, s->T[h].act, s->T[a].numel(),
                                     s->T[a].C, st);
          });
          break;
        }
        add("affine_fwd", 1, 0.0, 2 * tbytes(a), [=](cudaStream_t st) {
          fo::affine_fwd(act(a), P(s, i, 0), P(s, i, 1), s->T[o].act, s->T[a].rows(), s->T[a].C, dt, relu, st);
        });
        break;
      case FO_OP_RELU:
        add("relu_fwd", 1, 0.0, 2 * tbytes(a), [=](cudaStream_t st) {
          fo::relu_fwd(act(a), s->T[o].act, s->T[a].numel(), dt, st);
        });
        break;
      case FO_OP_MAXPOOL2:
        add("maxpool2_fwd", 1, 0.0, tbytes(a) + tbytes(o), [=](cudaStream_t st) {
          const Tensor& x = s->T[a];
          fo::maxpool2_fwd(act(a), s->T[o].act, x.N, x.H, x.W, x.C, dt, st);
        });
        break;
      case FO_OP_ADD: {
        const int b = op.in1;
        add("add_fwd", 1, 0.0, 3 * tbytes(i + 1), [=](cudaStream_t st) {
          fo::add_fwd(act(a), act(b), s->T[o].act, s->T[o].numel(), dt, relu, st);
        });
        break;
      }
      case FO_OP_AVGPOOL:
        add("avgpool_fwd", 1, 0.0, tbytes(a) + tbytes(o), [=](cudaStream_t st) {
          const Tensor& x = s->T[a];
          fo::avgpool_fwd(act(a), s->T[o].act, x.N, x.H * x.W, x.C, dt, st);
        });
        break;
      case FO_OP_FLATTEN:
        break;  // a view
      case FO_OP_LAYERNORM:
        add("layernorm_fwd", 1, 0.0, 2 * tbytes(a), [=](cudaStream_t st) {
          fo::layernorm_fwd(act(a), P(s, i, 0), P(s, i, 1), s->T[o].act, s->ln_mean[i], s->ln_rstd[i],
                            s->T[a].rows(), s->T[a].C, dt, st);
        });
        break;
      case FO_OP_GELU:
        if (gelu_done[i]) break;   // stored by the producing GEMM's epilogue
        add("gelu_fwd", 1, 0.0, 2 * tbytes(a), [=](cudaStream_t st) {
          fo::gelu_fwd(act(a), s->T[o].act, s->T[a].numel(), dt, st);
        });
        break;
      case FO_OP_ATTENTION: {
        const double Ls = ta.H, heads = op.heads, dh = double(op.cin) / op.heads;
        fo::AttnTcPlan* tp = nullptr;
        if (s->tc && dt == fo::kBF16 && !s->T[a].is_input() && !getenv("FO_NO_TC") && fo::attention_tc_ok(ta.H, op.cin, op.heads))
          tp = fo::attention_tc_plan(s->T[a].act, s->T[o].act, s->T[o].grad, ta.N, ta.H, op.cin, op.heads,
                                     fo::tc_error_word(s->tc));
        s->attn_tc[i] = tp;
        if (tp) {
          add("tc_attention_fwd", 1, 4.0 * ta.N * heads * Ls * Ls * dh, tbytes(a) + tbytes(o), [=](cudaStream_t st) {
            fo::attention_tc_fwd(tp, s->cur_len, s->T[o].act, s->attn_probs[i], s->T[a].N, st);
          });
          break;
        }
        add("attention_fwd", 1, 4.0 * ta.N * heads * Ls * Ls * dh, tbytes(a) + tbytes(o), [=](cudaStream_t st) {
          const Tensor& x = s->T[a];
          fo::attention_fwd(act(a), s->cur_len, s->T[o].act, s->attn_probs[i], x.N, x.H, op.cin, op.heads, dt, st);
        });
        break;
      }
      case FO_OP_MEANPOOL:
        add("meanpool_fwd", 1, 0.0, tbytes(a) + tbytes(o), [=](cudaStream_t st) {
          const Tensor& x = s->T[a];
          fo::meanpool_fwd(act(a), s->cur_len, s->T[o].act, x.N, x.H, x.C, dt, st);
        });
        break;
      case FO_OP_DWCONV: {
        const fo::DwShape d = dw_shape(s, i);
        add("dwconv_fwd", 1, 2.0 * double(to.numel()) * op.k * op.k, tbytes(a) + tbytes(o), [=](cudaStream_t st) {
          // the bf16 path multiplies the bf16 copy of the weights, like the convolutions
          const void* w = dt == fo::kBF16 ? (const void*)SH(s, i, 0) : (const void*)P(s, i, 0);
          fo::dwconv_fwd(d, act(a), w, op.bias ? P(s, i, 1) : nullptr, s->T[o].act, dt, st);
        });
        break;
      }
      case FO_OP_HSWISH:
        add("hswish_fwd", 1, 0.0, 2 * tbytes(a), [=](cudaStream_t st) {
          fo::hswish_fwd(act(a), s->T[o].act, s->T[a].numel(), dt, st);
        });
        break;
      case FO_OP_HSIGMOID:
        add("hsigmoid_fwd", 1, 0.0, 2 * tbytes(a), [=](cudaStream_t st) {
          fo::hsigmoid_fwd(act(a), s->T[o].act, s->T[a].numel(), dt, st);
        });
        break;
      case FO_OP_CHMUL: {
        const int b = op.in1;
        add("chmul_fwd", 1, 0.0, 2 * tbytes(a) + tbytes(b), [=](cudaStream_t st) {
          const Tensor& x = s->T[a];
          fo::chmul_fwd(act(a), act(b), s->T[o].act, x.N, x.H * x.W, x.C, dt, st);
        });
        break;
      }
    }
  }

  // ---------------- loss (softmax cross-entropy on fp32 logits)
  if (!fu.head) {
    const int lt = nops;
    add("softmax_ce", 1, 0.0, 2 * tbytes(lt), [=](cudaStream_t st) {
      fo::softmax_ce((const float*)s->T[lt].act, s->cur_labels, s->cfg.batch, s->cfg.num_classes, s->losses,
                     s->d_step, s->kLossRing - 1, s->T[lt].grad, fo::kF32, st);
    });
  }

  // ---------------- backward
  std::vector<char> written(nops + 1, 0);
  written[nops] = 1;  // dlogits
  // Contribution to tensor `tid`'s gradient: returns the accumulate flag
  // and marks the root written; tensor 0 receives none.
  // A fused residual add leaves the residual operand's first contribution
  // (the add's output gradient) pending: root -> tensor whose gradient is
  // still to be added.  The next contributor that can add it in its own
  // epilogue takes it as an addend; any other contributor, and any kernel
  // that reads the gradient, first has it copied in.
  std::vector<int> pending(nops + 1, -1);
  // Bias gradients from the kernel that writes the output gradient last: a
  // layernorm backward adds up the columns of what it stores as it goes
  // (partial sums per row block), which saves the bias pass a read of the
  // whole gradient.  Per gradient buffer (a fused residual's
  // branch shares the add output's), the request slot of its last writer,
  // or null when that writer cannot.
  struct PartReq {
    float* buf = nullptr;
    int chunks = 0;
  };
  std::vector<int> galias(nops + 1, -1);
  for (int i = 0; i < nops; ++i)
    if (fu.branch_of[i] >= 0) galias[fu.branch_of[i]] = i + 1;
  auto groot = [&](int tid) { return galias[tid] >= 0 ? s->T[galias[tid]].root : s->T[tid].root; };
  std::vector<std::shared_ptr<PartReq>> last_part(nops + 1);
  auto materialize = [&](int tid) {
    const int r = s->T[tid].root;
    if (pending[r] < 0) return;
    const int src = pending[r];
    pending[r] = -1;
    last_part[r] = nullptr;
    last_part[groot(tid)] = nullptr;
    const int64_t n = s->T[r].numel();
    add("add_bwd", 1, 0.0, 2 * tbytes(r), [=](cudaStream_t st) {
      fo::grad_split(s->T[src].grad, nullptr, s->T[r].grad, false, nullptr, false, n, dt, st);
    });
  };
  auto contrib = [&](int tid) -> int {
    materialize(tid);
    int r = s->T[tid].root;
    int accf = written[r] ? 1 : 0;
    written[r] = 1;
    last_part[groot(tid)] = nullptr;   // callers that store partials set their request after this
    return accf;
  };
  // A contribution whose kernel adds `*addend` (a pending gradient) itself.
  auto contrib_addend = [&](int tid, const void** addend) -> int {
    const int r = s->T[tid].root;
    *addend = nullptr;
    if (pending[r] >= 0) {
      *addend = s->T[pending[r]].grad;
      pending[r] = -1;
      last_part[groot(tid)] = nullptr;
      return 0;
    }
    return contrib(tid);
  };
  // Parameter-gradient reductions deferred to two batched launches after the
  // backward pass: column sums for the conv / linear biases, and the finish
  // of the affine / layernorm partials.  Each has its own partial buffer.
  std::vector<fo::ColsumTask> bias_tasks;
  std::vector<fo::FinishTask> finish_tasks;
  double deferred_bytes = 0.0;
  // Weight tensors whose optimizer update runs on the side stream as soon as
  // their gradient is complete and no kernel of the step reads them any more
  // (their layer's input gradient has run): the update's HBM traffic then
  // overlaps the rest of the backward pass.  Flags per 64 parameters.
  std::vector<uint8_t> early(size_t(s->n_padded / 64), 0);
  fo::SgdSegments group{};
  int64_t group_params = 0;
  auto flush_group = [&]() {
    if (group.n == 0) return;
    const fo::SgdSegments sg = group;
    add("sgd_momentum", 1, 0.0, double(sg.pre4[sg.n]) * 4.0 * (20.0 + (s->shadow ? 2.0 : 0.0)), [=](cudaStream_t st) {
      fo::sgd_momentum_segments(s->theta, s->mom, s->grad, s->shadow, sg, s->opt.lr, s->opt.momentum, st);
    }, 2);
    group = fo::SgdSegments{};
    group_params = 0;
  };
  for (int i = nops - 1; i >= 0; --i) {
    const fo_op op = s->ops[i];
    if (fu.skip_bwd[i]) {
      written[s->T[i + 1].root] = 1;
      continue;
    }
    if (fu.hswish_by[i] >= 0 || fu.relu_into_add[i] >= 0) {
      // the producer's backward applies this hard swish / relu: its input
      // gradient is present exactly when the output's is
      materialize(i + 1);   // the producer's backward reads this op's output gradient
      written[s->T[op.in0].root] = written[s->T[i + 1].root];
      continue;
    }
    const int a0 = op.in0, o = i + 1;
    const int ro = s->T[o].root;
    materialize(o);   // this op's backward reads its output gradient
    if (!written[ro]) {
      // Nothing downstream produced a gradient: zero this op's parameter grads.
      for (int si : s->op_segs[i]) {
        const ParamSeg seg = s->segs[si];
        add("memset_grad", 1, 0.0, seg.n * 4.0, [=](cudaStream_t st) {
          cudaMemsetAsync(s->grad + seg.off, 0, seg.n * sizeof(float), st);
        });
      }
      continue;
    }
    // A relu between this op's input and its producer: write the producer's
    // output gradient directly, masked by the relu output.
    const int mr = fu.bwd_mask[i];
    const int a = mr >= 0 ? s->ops[mr].in0 : a0;            // gradient destination
    const void* mask = mr >= 0 ? s->T[mr + 1].act : nullptr;
    const bool need_dx = !s->T[a0].is_input();
    const double csb = double(s->T[o].rows()) * s->T[o].C * esz;  // one read of dy
    if (fu.head && i == L) {
      const int B = s->cfg.batch, K = op.cin, C = op.cout;
      add("head_wgrad", 1, 2.0 * B * K * C, tbytes(a0), [=](cudaStream_t st) {
        fo::head_weight_grad((const float*)s->T[o].grad, act(a0), s->T[a0].dt, B, K, C, G(s, i, 0),
                             op.bias ? G(s, i, 1) : nullptr, s->row_loss, s->losses, s->d_step,
                             s->kLossRing - 1, st);
      }, 1);
      if (need_dx && contrib(a) != 0)   // formed in the forward launch as the first contribution
        return set_err(FO_ERR_ARG, "classifier input gradient is not the first contribution");
      continue;
    }
    switch (op.kind) {
      case FO_OP_CONV:
      case FO_OP_LINEAR: {
        fo::ConvShape cs = conv_shape(s, i);
        const int dto = s->T[o].dt, dta = s->T[a].dt;
        const bool bias = op.bias != 0;
        const double fl = 2.0 * double(s->T[o].rows()) * op.cout * double(op.kind == FO_OP_CONV ? op.k * op.k : 1) * op.cin;
        const std::shared_ptr<PartReq> lw = last_part[groot(o)];
        if (bias && lw && !lw->buf) {
          // the writer of this output gradient stores its column partials
          const Tensor& t = s->T[o];
          lw->buf = (float*)s->alloc(size_t(lw->chunks) * t.C * 4);
          if (!lw->buf) return set_err(FO_ERR_OOM, "bias-gradient partials");
          finish_tasks.push_back({lw->buf, G(s, i, 1), lw->chunks, t.C});
        } else if (bias && dto == fo::kBF16 && s->T[o].C % 8 == 0) {
          const Tensor& t = s->T[o];
          const int chunks = fo::colsum8_batch_chunks(t.rows());
          float* part = (float*)s->alloc(size_t(chunks) * t.C * 4);
          if (!part) return set_err(FO_ERR_OOM, "bias-gradient partials");
          bias_tasks.push_back({t.grad, part, t.rows(), t.C});
          finish_tasks.push_back({part, G(s, i, 1), chunks, t.C});
          deferred_bytes += double(t.bytes());
        } else if (bias) {
          add("bias_grad", 2, 0.0, double(s->T[o].bytes()), [=](cudaStream_t st) {
            fo::colsum(s->T[o].grad, nullptr, s->T[o].rows(), s->T[o].C, dto, s->colsum_scratch, G(s, i, 1), st,
                       true);
          });
        }
        // the weight gradient only feeds the optimizer: side stream, forked
        // before the input gradient so that the two run concurrently
        fo::TcGemm* tw = fo::tc_plan_wgrad(s->tc, s, i);
        if (tw) {
          add_tc(tw, 1);
        } else {
          const bool split = fo::simt_wgrad_splits(cs) > 1;
          add(op.kind == FO_OP_CONV ? "conv_wgrad_simt" : "linear_wgrad_simt", split ? 2 : 1, fl, 0.0,
              [=](cudaStream_t st) {
            fo::conv_wgrad_simt(cs, s->T[o].grad, dto, act(a0), s->T[a0].dt, G(s, i, 0),
                                split ? s->simt_scratch : nullptr, st);
          }, 1);
        }
        if (need_dx) {
          const void* addend = nullptr;
          const bool plain = fo::tc_plain_ok(s->tc, s, i);
          int accf = plain ? contrib_addend(a, &addend) : contrib(a);
          fo::TcEpilogue ex;
          ex.addend = addend;
          const bool fused = addend != nullptr;
          std::vector<fo::TcGemm*> tgs;
          bool zero_first = false;
          const bool planned = fo::tc_plan_dgrad(s->tc, s, i, accf, s->T[a].grad, mask, &tgs, &zero_first,
                                                 fused ? &ex : nullptr);
          if (fused && !planned)
            return set_err(FO_ERR_ARG, "op " + std::to_string(i) + ": fused input gradient not planned");
          if (planned) {
            if (zero_first) {
              const int ta = a;
              add("memset_dx", 1, 0.0, tbytes(ta), [=](cudaStream_t st) {
                cudaMemsetAsync(s->T[ta].grad, 0, s->T[ta].bytes(), st);
              });
            }
            for (fo::TcGemm* tg : tgs) add_tc(tg);
          } else {
            const bool wbf = dto == fo::kBF16;
            add(op.kind == FO_OP_CONV ? "conv_dgrad_simt" : "linear_dgrad_simt", 1, fl, 0.0, [=](cudaStream_t st) {
              const void* w = wbf ? (const void*)SH(s, i, 0) : (const void*)P(s, i, 0);
              fo::conv_dgrad_simt(cs, s->T[o].grad, dto, w, wbf ? fo::kBF16 : fo::kF32, s->T[a].grad, dta,
                                  accf != 0, mask, st);
            });
          }
        }
        if (s->segs[s->op_segs[i][0]].n >= kEarlyUpdateMin) {
          // the weights' update, after the input gradient that read them:
          // batched with the next weight tensors until the batch is large
          const ParamSeg seg = s->segs[s->op_segs[i][0]];
          const int64_t len = pad64(seg.n);
          group.off4[group.n] = seg.off / 4;
          group.pre4[group.n + 1] = group.pre4[group.n] + len / 4;
          ++group.n;
          group_params += len;
          for (int64_t b = seg.off / 64; b < (seg.off + len) / 64; ++b) early[size_t(b)] = 1;
          if (group_params >= kEarlyGroupMin || group.n == fo::kSgdMaxSegs) flush_group();
        }
        break;
      }
      case FO_OP_AFFINE:
        if (fo::vec8_ok(dt, s->T[a0].numel()) && s->T[a0].C % 8 == 0) {
          // one pass: dscale, dshift and dx (+)= dy * scale; behind a fused
          // hard swish, dy is formed from the hard swish's output gradient
          const int hs = fu.hswish_of[i];
          const int dyt = hs >= 0 ? hs + 1 : o;
          const int accf = need_dx ? contrib(a) : 0;
          const Tensor& x0 = s->T[a0];
          const int chunks = fo::affine_bwd8_chunks(x0.rows(), x0.C);
          float* ps = (float*)s->alloc(size_t(2) * chunks * x0.C * 4);
          if (!ps) return set_err(FO_ERR_OOM, "affine partials");
          float* ph = ps + size_t(chunks) * x0.C;
          finish_tasks.push_back({ps, G(s, i, 0), chunks, x0.C});
          finish_tasks.push_back({ph, G(s, i, 1), chunks, x0.C});
          add(hs >= 0 ? "affine_hswish_bwd" : "affine_bwd", 1, 0.0, (need_dx ? 3 + accf : 2) * csb + (hs >= 0) * csb,
              [=](cudaStream_t st) {
                const Tensor& x = s->T[a0];
                fo::affine_bwd8_pass(s->T[dyt].grad, act(a0), P(s, i, 0), need_dx ? s->T[a].grad : nullptr, accf != 0,
                                     x.rows(), x.C, ps, ph, st, hs >= 0 ? s->T[o].act : nullptr);
              });
          break;
        }
        add("affine_pgrad", 4, 0.0, 3 * csb, [=](cudaStream_t st) {
          const Tensor& x = s->T[a0];
          fo::colsum(s->T[o].grad, act(a0), x.rows(), x.C, dt, s->colsum_scratch, G(s, i, 0), st);
          fo::colsum(s->T[o].grad, nullptr, x.rows(), x.C, dt, s->colsum_scratch, G(s, i, 1), st);
        });
        if (need_dx) {
          int accf = contrib(a);
          add("affine_dx", 1, 0.0, (2 + accf) * csb, [=](cudaStream_t st) {
            fo::affine_dx(s->T[o].grad, P(s, i, 0), s->T[a].grad, s->T[a].rows(), s->T[a].C, dt, accf != 0, st);
          });
        }
        break;
      case FO_OP_RELU:
        if (need_dx) {
          int accf = contrib(a);
          // mask from the relu output: y > 0 exactly where x > 0
          add("relu_bwd", 1, 0.0, (3 + accf) * csb, [=](cudaStream_t st) {
            fo::relu_bwd(s->T[o].act, s->T[o].grad, s->T[a].grad, s->T[a].numel(), dt, accf != 0, st);
          });
        }
        break;
      case FO_OP_MAXPOOL2:
        if (need_dx && pool_codes[i]) {   // forward ran in the producing GEMM's epilogue
          int accf = contrib(a);
          const uint8_t* codes = pool_codes[i];
          add("relu_maxpool2_bwd", 1, 0.0, (2 + accf) * tbytes(a0) + 2.5 * csb, [=](cudaStream_t st) {
            const Tensor& x = s->T[a0];
            fo::relu_maxpool2_bwd_codes(s->T[o].act, codes, s->T[o].grad, s->T[a].grad, x.N, x.H, x.W, x.C,
                                        accf != 0, st);
          });
          break;
        }
        if (need_dx) {
          int accf = contrib(a);
          const bool masked = mr >= 0;
          add(masked ? "relu_maxpool2_bwd" : "maxpool2_bwd", 1, 0.0, (2 + accf) * tbytes(a0) + csb,
              [=](cudaStream_t st) {
                const Tensor& x = s->T[a0];
                if (masked)
                  fo::relu_maxpool2_bwd(act(a0), s->T[o].grad, s->T[a].grad, x.N, x.H, x.W, x.C, dt, accf != 0, st);
                else
                  fo::maxpool2_bwd(act(a0), s->T[o].grad, s->T[a].grad, x.N, x.H, x.W, x.C, dt, accf != 0, st);
              });
        }
        break;
      case FO_OP_ADD: {
        if (fu.branch_of[i] >= 0) {
          // the branch's gradient is this gradient (the same buffer); the
          // residual's is left pending for its next contributor
          written[s->T[fu.branch_of[i]].root] = 1;
          const int x = fu.add_other[i];
          if (s->T[x].is_input()) break;
          const int rx = s->T[x].root;
          if (!written[rx]) {
            pending[rx] = o;
            written[rx] = 1;
          } else {
            materialize(x);
            const int64_t n = s->T[o].numel();
            add("add_bwd", 1, 0.0, 3 * csb, [=](cudaStream_t st) {
              fo::grad_split(s->T[o].grad, nullptr, s->T[x].grad, true, nullptr, false, n, dt, st);
            });
          }
          break;
        }
        // one pass over the output gradient (masked by the relu after the
        // add when that relu's backward is folded in) into both inputs
        const int b = op.in1;
        const int rr = fu.add_relu[i];
        const int dyt = rr >= 0 ? rr + 1 : o;
        const void* msk = rr >= 0 ? s->T[rr + 1].act : nullptr;
        int srcs[2], accs[2], ns = 0;
        for (int src : {a0, b}) {
          if (s->T[src].is_input()) continue;
          srcs[ns] = src;
          accs[ns] = contrib(src);
          ++ns;
        }
        if (ns == 0) break;
        const int64_t n = s->T[o].numel();
        if (ns == 2 && s->T[srcs[0]].root == s->T[srcs[1]].root) {   // x + x: two passes into one buffer
          for (int q = 0; q < 2; ++q) {
            const int src = srcs[q], accf = accs[q];
            add("add_bwd", 1, 0.0, (2 + accf + (msk ? 1 : 0)) * csb, [=](cudaStream_t st) {
              fo::grad_split(s->T[dyt].grad, msk, s->T[src].grad, accf != 0, nullptr, false, n, dt, st);
            });
          }
          break;
        }
        const int s0 = srcs[0], s1 = ns == 2 ? srcs[1] : -1, acc0 = accs[0], acc1 = ns == 2 ? accs[1] : 0;
        add("add_bwd", 1, 0.0, (1 + (msk ? 1 : 0) + ns + acc0 + acc1) * csb, [=](cudaStream_t st) {
          fo::grad_split(s->T[dyt].grad, msk, s->T[s0].grad, acc0 != 0, s1 >= 0 ? s->T[s1].grad : nullptr,
                         acc1 != 0, n, dt, st);
        });
        break;
      }
      case FO_OP_AVGPOOL:
        if (need_dx) {
          int accf = contrib(a);
          add("avgpool_bwd", 1, 0.0, (1 + accf) * tbytes(a) + csb, [=](cudaStream_t st) {
            const Tensor& x = s->T[a];
            fo::avgpool_bwd(s->T[o].grad, x.grad, x.N, x.H * x.W, x.C, dt, accf != 0, st);
          });
        }
        break;
      case FO_OP_FLATTEN:
        break;  // shares the input's gradient buffer
      case FO_OP_LAYERNORM:
        if (fo::layernorm_bwd8_ok(dt, s->T[a0].C)) {
          const void* addend = nullptr;
          const int accf = need_dx ? contrib_addend(a, &addend) : 0;
          auto req = std::make_shared<PartReq>();
          req->chunks = fo::layernorm_bwd8_blocks(s->T[a0].rows());
          if (need_dx) last_part[groot(a)] = req;
          const Tensor& x0 = s->T[a0];
          const int blocks = fo::layernorm_bwd8_blocks(x0.rows());
          float* pg = (float*)s->alloc(size_t(2) * blocks * x0.C * 4);
          if (!pg) return set_err(FO_ERR_OOM, "layernorm partials");
          float* pb = pg + size_t(blocks) * x0.C;
          finish_tasks.push_back({pg, G(s, i, 0), blocks, x0.C});
          finish_tasks.push_back({pb, G(s, i, 1), blocks, x0.C});
          add("layernorm_bwd", 1, 0.0, (need_dx ? 3 + accf + (addend ? 1 : 0) : 2) * csb, [=](cudaStream_t st) {
            const Tensor& x = s->T[a0];
            fo::layernorm_bwd8_pass(act(a0), P(s, i, 0), s->ln_mean[i], s->ln_rstd[i], s->T[o].grad,
                                    need_dx ? s->T[a].grad : nullptr, x.rows(), x.C, accf != 0, pg, pb, st, addend,
                                    req->buf);
          });
          break;
        }
        add("layernorm_pgrad", 4, 0.0, 3 * csb, [=](cudaStream_t st) {
          const Tensor& x = s->T[a0];
          fo::colsum_lnx(s->T[o].grad, act(a0), s->ln_mean[i], s->ln_rstd[i], x.rows(), x.C, dt, s->colsum_scratch,
                         G(s, i, 0), st);
          fo::colsum(s->T[o].grad, nullptr, x.rows(), x.C, dt, s->colsum_scratch, G(s, i, 1), st);
        });
        if (need_dx) {
          int accf = contrib(a);
          add("layernorm_bwd", 1, 0.0, (3 + accf) * csb, [=](cudaStream_t st) {
            const Tensor& x = s->T[a];
            fo::layernorm_bwd_dx(act(a), P(s, i, 0), s->ln_mean[i], s->ln_rstd[i], s->T[o].grad, x.grad, x.rows(),
                                 x.C, dt, accf != 0, st);
          });
        }
        break;
      case FO_OP_GELU:
        if (need_dx) {
          int accf = contrib(a);
          add("gelu_bwd", 1, 0.0, (3 + accf) * csb, [=](cudaStream_t st) {
            fo::gelu_bwd(act(a), s->T[o].grad, s->T[a].grad, s->T[a].numel(), dt, accf != 0, st);
          });
        }
        break;
      case FO_OP_ATTENTION:
        if (need_dx) {
          int accf = contrib(a);
          const Tensor& ta = s->T[a];
          const double Ls = ta.H, heads = op.heads, dh = double(op.cin) / op.heads;
          if (fo::AttnTcPlan* tp = s->attn_tc[i]) {
            add("tc_attention_bwd", 1, 10.0 * ta.N * heads * Ls * Ls * dh, (2 + accf) * tbytes(a) + 2 * csb,
                [=](cudaStream_t st) {
                  fo::attention_tc_bwd(tp, s->cur_len, s->attn_probs[i], s->T[a].grad, s->T[a].N, accf != 0, st);
                });
            break;
          }
          add("attention_bwd", 1, 8.0 * ta.N * heads * Ls * Ls * dh, (2 + accf) * tbytes(a) + 2 * csb,
              [=](cudaStream_t st) {
                const Tensor& x = s->T[a];
                fo::attention_bwd(act(a), s->cur_len, s->attn_probs[i], s->T[o].act, s->T[o].grad, x.grad, x.N, x.H,
                                  op.cin, op.heads, dt, accf != 0, st);
              });
        }
        break;
      case FO_OP_MEANPOOL:
        if (need_dx) {
          int accf = contrib(a);
          add("meanpool_bwd", 1, 0.0, (1 + accf) * tbytes(a) + csb, [=](cudaStream_t st) {
            const Tensor& x = s->T[a];
            fo::meanpool_bwd(s->T[o].grad, s->cur_len, x.grad, x.N, x.H, x.C, dt, accf != 0, st);
          });
        }
        break;
      case FO_OP_DWCONV: {
        const fo::DwShape d = dw_shape(s, i);
        const int kk = op.k * op.k;
        const double fl = 2.0 * double(s->T[o].numel()) * kk;
        if (need_dx) {
          int accf = contrib(a);
          add("dwconv_dgrad", 1, fl, (1 + accf) * tbytes(a) + csb, [=](cudaStream_t st) {
            const void* w = dt == fo::kBF16 ? (const void*)SH(s, i, 0) : (const void*)P(s, i, 0);
            fo::dwconv_dgrad(d, s->T[o].grad, w, s->T[a].grad, dt, accf != 0, st);
          });
        }
        // weight (and bias) gradient partials, summed by the batched finish
        const int chunks = fo::dwconv_wgrad_chunks(d);
        float* pw = (float*)s->alloc(size_t(chunks) * op.cin * (kk + (op.bias ? 1 : 0)) * 4);
        if (!pw) return set_err(FO_ERR_OOM, "depthwise weight-gradient partials");
        float* pb = op.bias ? pw + size_t(chunks) * op.cin * kk : nullptr;
        finish_tasks.push_back({pw, G(s, i, 0), chunks, op.cin * kk});
        if (pb) finish_tasks.push_back({pb, G(s, i, 1), chunks, op.cin});
        add("dwconv_wgrad", 1, fl, tbytes(a0) + csb, [=](cudaStream_t st) {
          fo::dwconv_wgrad_pass(d, s->T[o].grad, act(a0), dt, pw, pb, st);
        });
        break;
      }
      case FO_OP_HSWISH:
        if (need_dx) {
          int accf = contrib(a);
          add("hswish_bwd", 1, 0.0, (3 + accf) * csb, [=](cudaStream_t st) {
            fo::hswish_bwd(act(a0), s->T[o].grad, s->T[a].grad, s->T[a].numel(), dt, accf != 0, st);
          });
        }
        break;
      case FO_OP_HSIGMOID:
        if (need_dx) {
          int accf = contrib(a);
          add("hsigmoid_bwd", 1, 0.0, (3 + accf) * csb, [=](cudaStream_t st) {
            fo::hsigmoid_bwd(act(a0), s->T[o].grad, s->T[a].grad, s->T[a].numel(), dt, accf != 0, st);
          });
        }
        break;
      case FO_OP_CHMUL: {
        const int b = op.in1;
        const int acc_dx = need_dx ? contrib(a0) : 0;
        const bool need_ds = b != 0;
        const int acc_ds = need_ds ? contrib(b) : 0;
        add("chmul_bwd", 1, 0.0, (2 + (need_dx ? 1 + acc_dx : 0)) * csb + (1 + acc_ds) * tbytes(b),
            [=](cudaStream_t st) {
              const Tensor& x = s->T[a0];
              fo::chmul_bwd(act(a0), act(b), s->T[o].grad, need_dx ? s->T[a0].grad : nullptr, acc_dx != 0,
                            need_ds ? s->T[b].grad : nullptr, acc_ds != 0, x.N, x.H * x.W, x.C, dt, st);
            });
        break;
      }
    }
  }

  for (int r = 0; r <= nops; ++r) materialize(r);
  flush_group();

  // ---------------- optimizer (Algorithm 4: theta_s <- theta_s - gamma_s * update)
  if (!bias_tasks.empty())
    add("bias_grad", int((bias_tasks.size() + 39) / 40), 0.0, deferred_bytes, [=](cudaStream_t st) {
      fo::colsum8_batched(bias_tasks, st);
    });
  if (!finish_tasks.empty()) {
    double fb = 0.0;
    for (const fo::FinishTask& t : finish_tasks) fb += 4.0 * double(t.chunks + 1) * t.C;
    add("param_grad_finish", int((finish_tasks.size() + 39) / 40), 0.0, fb, [=](cudaStream_t st) {
      fo::finish_batched(finish_tasks, st);
    });
  }
  // the final update covers the parameters not updated early: the whole
  // vector, a list of 64-element blocks when that list is short, or the
  // whole vector minus flagged blocks
  std::vector<int64_t> late;
  for (size_t b = 0; b < early.size(); ++b)
    if (!early[b]) late.push_back(int64_t(b));
  const double late_bytes = double(late.size()) * 64.0 * (20.0 + (s->shadow ? 2.0 : 0.0));
  if (late.size() == early.size()) {
    add("sgd_momentum", 1, 0.0, late_bytes, [=](cudaStream_t st) {
      fo::sgd_momentum(s->theta, s->mom, s->grad, s->shadow, s->n_padded, s->opt.lr, s->opt.momentum, s->d_step, st);
    });
  } else if (late.size() * 8 < early.size()) {
    int64_t* blk = (int64_t*)s->alloc(std::max<size_t>(late.size(), 1) * sizeof(int64_t));
    if (!blk) return set_err(FO_ERR_OOM, "optimizer block list");
    if (!late.empty()) FO_CUDA(cudaMemcpy(blk, late.data(), late.size() * sizeof(int64_t), cudaMemcpyHostToDevice));
    const int64_t nb = int64_t(late.size());
    add("sgd_momentum", 1, 0.0, late_bytes, [=](cudaStream_t st) {
      fo::sgd_momentum_blocks(s->theta, s->mom, s->grad, s->shadow, blk, nb, s->opt.lr, s->opt.momentum, s->d_step,
                              st);
    });
  } else {
    uint8_t* skip = (uint8_t*)s->alloc(early.size());
    if (!skip) return set_err(FO_ERR_OOM, "optimizer flags");
    FO_CUDA(cudaMemcpy(skip, early.data(), early.size(), cudaMemcpyHostToDevice));
    add("sgd_momentum", 1, 0.0, late_bytes, [=](cudaStream_t st) {
      fo::sgd_momentum(s->theta, s->mom, s->grad, s->shadow, s->n_padded, s->opt.lr, s->opt.momentum, s->d_step,
                       st, skip);
    });
  }
  plan.back().join = true;   // the side and optimizer streams join before the final update
  for (int i = 0; i < nops; ++i)
    if (s->ops[i].kind == FO_OP_ATTENTION) fo::attention_prepare(s->T[s->ops[i].in0].H, s->ops[i].cin, s->ops[i].heads);
  return FO_OK;
}

int allocate(fo_server* s) {
  const fo_server_cfg& c = s->cfg;
  size_t esz = s->dt == fo::kF32 ? 4 : 2;
  // parameters
  s->theta = (float*)s->alloc(s->n_padded * 4);
  s->mom = (float*)s->alloc(s->n_padded * 4);
  s->grad = (float*)s->alloc(s->n_padded * 4);
  if (!s->theta || !s->mom || !s->grad) return set_err(FO_ERR_OOM, "parameter allocation");
  FO_CUDA(cudaMemset(s->theta, 0, s->n_padded * 4));
  FO_CUDA(cudaMemset(s->mom, 0, s->n_padded * 4));
  FO_CUDA(cudaMemset(s->grad, 0, s->n_padded * 4));
  if (s->dt == fo::kBF16) {
    s->shadow = (fo::bf16*)s->alloc(s->n_padded * 2);
    if (!s->shadow) return set_err(FO_ERR_OOM, "shadow allocation");
    FO_CUDA(cudaMemset(s->shadow, 0, s->n_padded * 2));
  }
  // activation slab: omega slots (Eq. 3), 256-byte aligned each
  s->slot_act_bytes = int64_t(c.batch) * c.in_h * c.in_w * c.in_c * esz;
  s->slot_stride = (s->slot_act_bytes + 255) / 256 * 256;
  s->slab = (char*)s->alloc(size_t(s->slot_stride) * c.omega);
  s->slot_labels = (int32_t*)s->alloc(size_t(c.omega) * c.batch * 4);
  s->slot_lengths = (int32_t*)s->alloc(size_t(c.omega) * c.batch * 4);
  if (!s->slab || !s->slot_labels || !s->slot_lengths) return set_err(FO_ERR_OOM, "activation slab");
  s->slot_ready.assign(c.omega, nullptr);
  s->slot_free.assign(c.omega, nullptr);
  s->slot_consumed.assign(c.omega, 0);
  for (int i = 0; i < c.omega; ++i) {
    FO_CUDA(cudaEventCreateWithFlags(&s->slot_ready[i], cudaEventDisableTiming));
    FO_CUDA(cudaEventCreateWithFlags(&s->slot_free[i], cudaEventDisableTiming));
  }
  s->stage_stride = (s->slot_stride + 2 * int64_t(c.batch) * 4 + 255) / 256 * 256;
  s->stage_buf = (char*)s->alloc(size_t(s->stage_stride) * fo_server::kStage);
  if (!s->stage_buf) return set_err(FO_ERR_OOM, "upload staging");
  s->stage_landed.assign(fo_server::kStage, nullptr);
  s->stage_free.assign(fo_server::kStage, nullptr);
  for (int r = 0; r < fo_server::kStage; ++r) {
    FO_CUDA(cudaEventCreateWithFlags(&s->stage_landed[r], cudaEventDisableTiming));
    FO_CUDA(cudaEventCreateWithFlags(&s->stage_free[r], cudaEventDisableTiming));
  }
  s->step_done.assign(fo_server::kStepEvents, nullptr);
  for (cudaEvent_t& e : s->step_done) FO_CUDA(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
  // tensors
  int nops = int(s->ops.size());
  for (int tid = 1; tid <= nops; ++tid) {
    Tensor& t = s->T[tid];
    if (t.root != tid) continue;
    t.act = s->alloc(t.bytes());
    t.grad = s->alloc(t.bytes());
    if (!t.act || !t.grad) return set_err(FO_ERR_OOM, "tensor allocation");
  }
  for (int tid = 1; tid <= nops; ++tid) {
    Tensor& t = s->T[tid];
    if (t.root != tid) {
      t.act = s->T[t.root].act;
      t.grad = s->T[t.root].grad;
    }
  }
  // scratch for deterministic column sums
  int64_t cs_floats = 1;
  for (int i = 0; i < nops; ++i) {
    const Tensor& o = s->T[i + 1];
    const Tensor& a = s->T[s->ops[i].in0];
    cs_floats = std::max(cs_floats, fo::server_colsum_floats(o.rows(), o.C));
    cs_floats = std::max(cs_floats, fo::server_colsum_floats(a.rows(), a.C));
  }
  s->colsum_scratch = (float*)s->alloc(cs_floats * 4);
  int64_t simt_floats = 0;   // split-K partials of the CUDA-core weight gradient
  for (int i = 0; i < nops; ++i)
    if (s->ops[i].kind == FO_OP_CONV || s->ops[i].kind == FO_OP_LINEAR)
      simt_floats = std::max(simt_floats, fo::simt_wgrad_scratch_floats(conv_shape(s, i)));
  s->simt_scratch = simt_floats ? (float*)s->alloc(simt_floats * 4) : nullptr;
  s->ln_mean.assign(nops, nullptr);
  s->ln_rstd.assign(nops, nullptr);
  s->attn_probs.assign(nops, nullptr);
  for (int i = 0; i < nops; ++i) {
    const fo_op& op = s->ops[i];
    const Tensor& a = s->T[op.in0];
    if (op.kind == FO_OP_LAYERNORM) {
      s->ln_mean[i] = (float*)s->alloc(a.rows() * 4);
      s->ln_rstd[i] = (float*)s->alloc(a.rows() * 4);
    } else if (op.kind == FO_OP_ATTENTION) {
      s->attn_probs[i] = (float*)s->alloc(size_t(a.N) * op.heads * a.H * a.H * 4);
    }
  }
  s->losses = (float*)s->alloc(size_t(s->kLossRing) * 4);
  s->row_loss = (float*)s->alloc(size_t(s->cfg.batch) * 4);
  s->d_step = (int64_t*)s->alloc(sizeof(int64_t));
  if (!s->row_loss || !s->d_step) return set_err(FO_ERR_OOM, "scratch allocation");
  FO_CUDA(cudaMemset(s->d_step, 0, sizeof(int64_t)));
  s->graphs.assign(s->cfg.omega, nullptr);
  s->prof_graphs.assign(s->cfg.omega, nullptr);
  s->prof_events.assign(s->cfg.omega, {});
  s->use_graphs = getenv("FO_NO_GRAPH") == nullptr;
  if (!s->colsum_scratch || !s->losses) return set_err(FO_ERR_OOM, "scratch allocation");
  FO_CUDA(cudaMemset(s->losses, 0, size_t(s->kLossRing) * 4));
  return FO_OK;
}

void destroy_impl(fo_server* s) {
  if (!s) return;
  if (s->cs) cudaStreamSynchronize(s->cs);
  if (s->as) cudaStreamSynchronize(s->as);
  for (fo::AttnTcPlan* a : s->attn_tc) fo::attention_tc_destroy(a);
  s->attn_tc.clear();
  if (s->xs) cudaStreamSynchronize(s->xs);
  if (s->hs) cudaStreamSynchronize(s->hs);
  for (auto g : s->graphs) if (g) cudaGraphExecDestroy(g);
  for (auto g : s->prof_graphs) if (g) cudaGraphExecDestroy(g);
  for (auto& v : s->prof_events)
    for (auto& r : v) {
      cudaEventDestroy(r.a);
      cudaEventDestroy(r.b);
    }
  fo::tc_destroy(s->tc);
  for (auto e : s->slot_ready) if (e) cudaEventDestroy(e);
  for (auto e : s->slot_free) if (e) cudaEventDestroy(e);
  for (auto e : s->step_done) if (e) cudaEventDestroy(e);
  for (auto& r : s->prof) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (auto e : s->ev_pool) cudaEventDestroy(e);
  if (s->side) cudaStreamSynchronize(s->side);
  if (s->opt_st) cudaStreamSynchronize(s->opt_st);
  for (void* p : s->allocs) cudaFree(p);
  for (int b = 0; b < 2; ++b) {
    if (s->agg_stage[b]) cudaFree(s->agg_stage[b]);
    if (s->agg_landed[b]) cudaEventDestroy(s->agg_landed[b]);
    if (s->agg_read[b]) cudaEventDestroy(s->agg_read[b]);
  }
  if (s->cs) cudaStreamDestroy(s->cs);
  if (s->as) cudaStreamDestroy(s->as);
  if (s->agg_ev) cudaEventDestroy(s->agg_ev);
  if (s->xs) cudaStreamDestroy(s->xs);
  if (s->hs) cudaStreamDestroy(s->hs);
  for (auto e : s->stage_landed) if (e) cudaEventDestroy(e);
  for (auto e : s->stage_free) if (e) cudaEventDestroy(e);
  if (s->side) cudaStreamDestroy(s->side);
  if (s->opt_st) cudaStreamDestroy(s->opt_st);
  if (s->fork2_ev) cudaEventDestroy(s->fork2_ev);
  if (s->join2_ev) cudaEventDestroy(s->join2_ev);
  if (s->fork_ev) cudaEventDestroy(s->fork_ev);
  if (s->join_ev) cudaEventDestroy(s->join_ev);
  delete s->sched;
  delete s;
}

int prof_id(fo_server* s, const char* name) {
  for (size_t q = 0; q < s->prof_names.size(); ++q)
    if (std::strcmp(s->prof_names[q], name) == 0) return int(q);
  s->prof_names.push_back(name);
  return int(s->prof_names.size()) - 1;
}

// Capture the step plan for batch slot `slot` into an executable graph.
int capture_slot(fo_server* s, int slot, cudaGraphExec_t* out) {
  const int B = s->cfg.batch;
  s->cur_in = s->slab + size_t(slot) * s->slot_stride;
  s->cur_labels = s->slot_labels + size_t(slot) * B;
  s->cur_len = s->slot_lengths + size_t(slot) * B;
  fo::tc_set_input(s->tc, slot);
  cudaGraph_t g = nullptr;
  FO_CUDA(cudaStreamBeginCapture(s->cs, cudaStreamCaptureModeRelaxed));
  bool forked = false, forked2 = false;
  for (const Launch& l : s->plan) {
    if (l.join && forked) {
      FO_CUDA(cudaEventRecord(s->join_ev, s->side));
      FO_CUDA(cudaStreamWaitEvent(s->cs, s->join_ev, 0));
      forked = false;
    }
    if (l.join && forked2) {
      FO_CUDA(cudaEventRecord(s->join2_ev, s->opt_st));
      FO_CUDA(cudaStreamWaitEvent(s->cs, s->join2_ev, 0));
      forked2 = false;
    }
    if (l.lane == 2 && s->use_side) {
      // after the compute stream's work so far and the side stream's
      FO_CUDA(cudaEventRecord(s->fork_ev, s->cs));
      FO_CUDA(cudaStreamWaitEvent(s->opt_st, s->fork_ev, 0));
      if (forked) {
        FO_CUDA(cudaEventRecord(s->fork2_ev, s->side));
        FO_CUDA(cudaStreamWaitEvent(s->opt_st, s->fork2_ev, 0));
      }
      forked2 = true;
      l.fn(s->opt_st);
      continue;
    }
    if (l.lane == 1 && s->use_side) {
      // fork after everything the compute stream has issued so far
      FO_CUDA(cudaEventRecord(s->fork_ev, s->cs));
      FO_CUDA(cudaStreamWaitEvent(s->side, s->fork_ev, 0));
      forked = true;
      l.fn(s->side);
    } else {
      l.fn(s->cs);
    }
  }
  if (forked) {
    FO_CUDA(cudaEventRecord(s->join_ev, s->side));
    FO_CUDA(cudaStreamWaitEvent(s->cs, s->join_ev, 0));
  }
  if (forked2) {
    FO_CUDA(cudaEventRecord(s->join2_ev, s->opt_st));
    FO_CUDA(cudaStreamWaitEvent(s->cs, s->join2_ev, 0));
  }
  FO_CUDA(cudaStreamEndCapture(s->cs, &g));
  cudaError_t e = cudaGraphInstantiate(out, g, 0);
  cudaGraphDestroy(g);
  if (e != cudaSuccess) return set_err(FO_ERR_CUDA, std::string("graph instantiate: ") + cudaGetErrorString(e));
  return FO_OK;
}

cudaEvent_t pool_event(fo_server* s) {
  if (!s->ev_pool.empty()) {
    cudaEvent_t e = s->ev_pool.back();
    s->ev_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

}  // namespace

// ===================================================================== C ABI

extern "C" {

const char* fo_last_error(void) { return g_err.c_str(); }

static int server_create(const fo_op* ops, int n_ops, const fo_optimizer* opt, const fo_server_cfg* cfg,
                         fo_server** out, fo_server** held);

// No C++ exception crosses the C ABI: a host allocation that fails inside
// (std::bad_alloc) releases the half-built server and returns FO_ERR_OOM.
int fo_server_create(const fo_op* ops, int n_ops, const fo_optimizer* opt, const fo_server_cfg* cfg,
                     fo_server** out) {
  fo_server* held = nullptr;
  try {
    return server_create(ops, n_ops, opt, cfg, out, &held);
  } catch (const std::bad_alloc&) {
    destroy_impl(held);
    return set_err(FO_ERR_OOM, "host allocation");
  } catch (const std::exception& e) {
    destroy_impl(held);
    return set_err(FO_ERR_ARG, e.what());
  }
}

static int server_create(const fo_op* ops, int n_ops, const fo_optimizer* opt, const fo_server_cfg* cfg,
                         fo_server** out, fo_server** held) {
  g_err.clear();
  if (!ops || n_ops <= 0 || !opt || !cfg || !out) return set_err(FO_ERR_ARG, "null argument");
  *out = nullptr;
  const fo_server_cfg& c = *cfg;
  if (c.num_devices <= 0 || c.num_devices > FO_MAX_DEVICES || c.omega <= 0 || c.omega > FO_MAX_OMEGA ||
      c.depth <= 0 || c.batch <= 0 || c.batch > 1024 ||
      c.in_h <= 0 || c.in_w <= 0 || c.in_c <= 0 || c.num_classes <= 0 ||
      (c.dtype != FO_DTYPE_F32 && c.dtype != FO_DTYPE_BF16) || c.max_delay < 0 ||
      (c.sched_policy != FO_SCHED_COUNTER && c.sched_policy != FO_SCHED_FIFO))
    return set_err(FO_ERR_ARG, "bad server configuration");
  if (int64_t(c.in_h) * c.in_w * c.in_c > INT32_MAX)
    return set_err(FO_ERR_ARG, "more than 2^31 - 1 activation elements per sample");
  fo_server* s = new (std::nothrow) fo_server();
  if (!s) return set_err(FO_ERR_OOM, "host allocation");
  *held = s;
  s->cfg = c;
  s->opt = *opt;
  s->dt = c.dtype == FO_DTYPE_F32 ? fo::kF32 : fo::kBF16;
  s->ops.assign(ops, ops + n_ops);
  int rc = infer(s);
  if (rc != FO_OK) {
    destroy_impl(s);
    return rc;
  }
  s->sched = new fo::TaskScheduler(c.num_devices, c.omega, c.depth, c.sched_policy);
  s->use_side = getenv("FO_NO_SIDE") == nullptr;
  if (cudaStreamCreateWithFlags(&s->cs, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&s->xs, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&s->hs, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&s->side, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&s->opt_st, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&s->as, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&s->agg_ev, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&s->fork2_ev, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&s->join2_ev, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&s->fork_ev, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&s->join_ev, cudaEventDisableTiming) != cudaSuccess) {
    destroy_impl(s);
    return set_err(FO_ERR_CUDA, "stream creation");
  }
  rc = allocate(s);
  if (rc == FO_OK) rc = fo::tc_create(&s->tc, s);
  if (rc == FO_OK) rc = build_plan(s);
  if (rc == FO_OK) rc = fo::tc_finalize(s->tc);
  // Instantiate the step graph of every batch slot up front.
  for (int sl = 0; rc == FO_OK && s->use_graphs && sl < c.omega; ++sl) rc = capture_slot(s, sl, &s->graphs[sl]);
  if (rc == FO_OK && cudaDeviceSynchronize() != cudaSuccess) rc = set_err(FO_ERR_CUDA, "create sync");
  if (rc != FO_OK) {
    destroy_impl(s);
    return rc;
  }
  *out = s;
  return FO_OK;
}

int fo_server_destroy(fo_server* s) {
  destroy_impl(s);
  return FO_OK;
}

int64_t fo_server_num_params(const fo_server* s) { return s ? s->n_params : -1; }

static int copy_params(fo_server* s, float* dev, const float* host, float* host_out, int64_t n) {
  if (!s || n != s->n_params || (!host && !host_out)) return set_err(FO_ERR_ARG, "bad parameter vector");
  FO_CUDA(cudaStreamSynchronize(s->cs));
  for (const ParamSeg& g : s->segs) {
    if (host) FO_CUDA(cudaMemcpy(dev + g.off, host + g.flat, g.n * 4, cudaMemcpyHostToDevice));
    else FO_CUDA(cudaMemcpy(host_out + g.flat, dev + g.off, g.n * 4, cudaMemcpyDeviceToHost));
  }
  return FO_OK;
}

int fo_server_set_params(fo_server* s, const float* host, int64_t n) {
  int rc = copy_params(s, s ? s->theta : nullptr, host, nullptr, n);
  if (rc != FO_OK) return rc;
  if (s->shadow) {
    fo::f32_to_bf16(s->theta, s->shadow, s->n_padded, s->cs);
    FO_CUDA(cudaStreamSynchronize(s->cs));
  }
  return FO_OK;
}
int fo_server_get_params(fo_server* s, float* host, int64_t n) {
  return copy_params(s, s ? s->theta : nullptr, nullptr, host, n);
}
int fo_server_set_momentum(fo_server* s, const float* host, int64_t n) {
  return copy_params(s, s ? s->mom : nullptr, host, nullptr, n);
}
int fo_server_get_momentum(fo_server* s, float* host, int64_t n) {
  return copy_params(s, s ? s->mom : nullptr, nullptr, host, n);
}

int fo_server_tensor(const fo_server* s, int index, const void** data, int64_t* dims4, int* dtype) {
  if (!s || !data || !dims4 || !dtype) return set_err(FO_ERR_ARG, "null argument");
  if (index < 1 || index > int(s->ops.size())) return set_err(FO_ERR_ARG, "tensor index outside 1..n_ops");
  const Tensor& t = s->T[index];
  *data = t.is_input() ? s->cur_in : t.act;
  dims4[0] = t.N;
  dims4[1] = t.H;
  dims4[2] = t.W;
  dims4[3] = t.C;
  *dtype = t.dt;
  return FO_OK;
}

int fo_server_params_device(fo_server* s, float** theta, int64_t* n) {
  if (!s || !theta || !n) return set_err(FO_ERR_ARG, "null argument");
  *theta = s->theta;
  *n = s->n_padded;
  return FO_OK;
}

int fo_server_load_params_device(fo_server* s, const float* src, int64_t n) {
  if (!s || !src) return set_err(FO_ERR_ARG, "null argument");
  if (n != s->n_padded) return set_err(FO_ERR_ARG, "parameter vector length is not the padded length");
  FO_CUDA(cudaMemcpyAsync(s->theta, src, size_t(n) * 4, cudaMemcpyDeviceToDevice, s->cs));
  if (s->shadow) fo::f32_to_bf16(s->theta, s->shadow, s->n_padded, s->cs);
  return FO_OK;
}

int fo_server_store_params_device(fo_server* s, float* dst, int64_t n) {
  if (!s || !dst) return set_err(FO_ERR_ARG, "null argument");
  if (n != s->n_padded) return set_err(FO_ERR_ARG, "parameter vector length is not the padded length");
  FO_CUDA(cudaMemcpyAsync(dst, s->theta, size_t(n) * 4, cudaMemcpyDeviceToDevice, s->cs));
  return FO_OK;
}

// The copies of an accepted upload into batch slot `slot` (before the
// scheduler commits it).
static int upload_copies(fo_server* s, int32_t slot, const void* acts, const int32_t* labels,
                         const int32_t* lengths) {
  const int B = s->cfg.batch;
  char* d_act = s->slab + size_t(slot) * s->slot_stride;
  int32_t* d_lab = s->slot_labels + size_t(slot) * B;
  int32_t* d_len = s->slot_lengths + size_t(slot) * B;
  bool busy = false;   // a queued step still reads this slot
  if (s->slot_consumed[slot]) {
    const cudaError_t q = cudaEventQuery(s->slot_free[slot]);
    if (q == cudaErrorNotReady) busy = true;
    else FO_CUDA(q);
  }
  if (!busy) {
    FO_CUDA(cudaMemcpyAsync(d_act, acts, s->slot_act_bytes, cudaMemcpyDefault, s->hs));
    FO_CUDA(cudaMemcpyAsync(d_lab, labels, B * 4, cudaMemcpyDefault, s->hs));
    if (lengths) FO_CUDA(cudaMemcpyAsync(d_len, lengths, B * 4, cudaMemcpyDefault, s->hs));
    FO_CUDA(cudaEventRecord(s->slot_ready[slot], s->hs));
    // The caller may reuse its buffers once the call returns.
    FO_CUDA(cudaEventSynchronize(s->slot_ready[slot]));
    return FO_OK;
  }
  const int r = int(s->stage_next++ % fo_server::kStage);
  char* st = s->stage_buf + size_t(r) * s->stage_stride;
  int32_t* st_lab = reinterpret_cast<int32_t*>(st + s->slot_stride);
  int32_t* st_len = st_lab + B;
  FO_CUDA(cudaStreamWaitEvent(s->hs, s->stage_free[r], 0));   // the move that last read this buffer
  FO_CUDA(cudaMemcpyAsync(st, acts, s->slot_act_bytes, cudaMemcpyDefault, s->hs));
  FO_CUDA(cudaMemcpyAsync(st_lab, labels, B * 4, cudaMemcpyDefault, s->hs));
  if (lengths) FO_CUDA(cudaMemcpyAsync(st_len, lengths, B * 4, cudaMemcpyDefault, s->hs));
  FO_CUDA(cudaEventRecord(s->stage_landed[r], s->hs));
  FO_CUDA(cudaStreamWaitEvent(s->xs, s->stage_landed[r], 0));
  FO_CUDA(cudaStreamWaitEvent(s->xs, s->slot_free[slot], 0));
  FO_CUDA(cudaMemcpyAsync(d_act, st, s->slot_act_bytes, cudaMemcpyDeviceToDevice, s->xs));
  FO_CUDA(cudaMemcpyAsync(d_lab, st_lab, B * 4, cudaMemcpyDeviceToDevice, s->xs));
  if (lengths) FO_CUDA(cudaMemcpyAsync(d_len, st_len, B * 4, cudaMemcpyDeviceToDevice, s->xs));
  FO_CUDA(cudaEventRecord(s->stage_free[r], s->xs));
  FO_CUDA(cudaEventRecord(s->slot_ready[slot], s->xs));
  // The caller may reuse its buffers once its own copy is done.
  FO_CUDA(cudaEventSynchronize(s->stage_landed[r]));
  return FO_OK;
}

int fo_enqueue_activations(fo_server* s, int device_id, const void* acts, const int32_t* labels,
                           const int32_t* lengths, int* sender_on) {
  if (!s || !acts || !labels) return set_err(FO_ERR_ARG, "null argument");
  if (s->cfg.seq && !lengths) return set_err(FO_ERR_ARG, "lengths required for sequence batches");
  if (device_id < 0 || device_id >= s->cfg.num_devices) return set_err(FO_ERR_ARG, "bad device id");
  // The slot is filled first and the upload committed to Q^act_k only once
  // its copies are issued: a failed copy leaves the scheduler as it was.
  int32_t slot = -1;
  const int peek = s->sched->peek(device_id, &slot);
  if (peek == 0) {
    const int rc = upload_copies(s, slot, acts, labels, lengths);
    if (rc != FO_OK) {
      if (sender_on) *sender_on = s->sched->sender_on()[device_id];
      return rc;
    }
  }
  int32_t committed = -1;
  const int rc = s->sched->put(device_id, &committed);
  if (sender_on) *sender_on = s->sched->sender_on()[device_id];
  if (rc == -1) return set_err(FO_ERR_ARG, "device has left");
  if (rc == 2) return FO_FULL;
  if (committed != slot) return set_err(FO_ERR_ARG, "scheduler slot changed between peek and put");
  return FO_OK;
}

int fo_server_step(fo_server* s, int* device_used, int32_t* slot_used) {
  if (!s) return set_err(FO_ERR_ARG, "null server");
  int k = -1;
  int32_t slot = -1;
  if (s->sched->get(&k, &slot) != 0) {
    if (device_used) *device_used = -1;
    if (slot_used) *slot_used = -1;
    s->last_launches = 0;
    return FO_EMPTY;
  }
  if (device_used) *device_used = k;
  if (slot_used) *slot_used = slot;
  const int B = s->cfg.batch;
  s->cur_in = s->slab + size_t(slot) * s->slot_stride;
  s->cur_labels = s->slot_labels + size_t(slot) * B;
  s->cur_len = s->slot_lengths + size_t(slot) * B;
  fo::tc_set_input(s->tc, slot);
  FO_CUDA(cudaStreamWaitEvent(s->cs, s->slot_ready[slot], 0));
  int n = 0;
  for (const Launch& l : s->plan) n += l.kernels;
  if (!s->use_graphs) {
    for (const Launch& l : s->plan) {
      if (s->profiling) {
        ProfRec r{prof_id(s, l.name), pool_event(s), pool_event(s), l.kernels, l.flops, l.bytes};
        cudaEventRecord(r.a, s->cs);
        l.fn(s->cs);
        cudaEventRecord(r.b, s->cs);
        s->prof.push_back(r);
      } else {
        l.fn(s->cs);
      }
    }
  } else if (!s->profiling) {
    // One CUDA graph per batch slot: the slot's address and tensor maps are
    // the only per-step inputs the kernels take from the host.
    cudaGraphExec_t& ge = s->graphs[slot];
    if (!ge) {
      int rc = capture_slot(s, slot, &ge);
      if (rc != FO_OK) return rc;
    }
    FO_CUDA(cudaGraphLaunch(ge, s->cs));
  } else {
    // Profiled graph: event records around every plan entry, read back
    // after the step (no host launch gaps inside the step).
    cudaGraphExec_t& ge = s->prof_graphs[slot];
    std::vector<ProfRec>& evs = s->prof_events[slot];
    if (!ge) {
      evs.clear();
      cudaGraph_t g = nullptr;
      FO_CUDA(cudaStreamBeginCapture(s->cs, cudaStreamCaptureModeRelaxed));
      for (const Launch& l : s->plan) {
        ProfRec r{prof_id(s, l.name), nullptr, nullptr, l.kernels, l.flops, l.bytes};
        cudaEventCreate(&r.a);
        cudaEventCreate(&r.b);
        // External records become event nodes of the graph (timing events).
        FO_CUDA(cudaEventRecordWithFlags(r.a, s->cs, cudaEventRecordExternal));
        l.fn(s->cs);
        FO_CUDA(cudaEventRecordWithFlags(r.b, s->cs, cudaEventRecordExternal));
        evs.push_back(r);
      }
      FO_CUDA(cudaStreamEndCapture(s->cs, &g));
      cudaError_t e = cudaGraphInstantiate(&ge, g, 0);
      cudaGraphDestroy(g);
      if (e != cudaSuccess) return set_err(FO_ERR_CUDA, std::string("graph instantiate: ") + cudaGetErrorString(e));
    }
    FO_CUDA(cudaGraphLaunch(ge, s->cs));
    FO_CUDA(cudaStreamSynchronize(s->cs));
    for (const ProfRec& r : evs) {
      float t = 0.f;
      FO_CUDA(cudaEventElapsedTime(&t, r.a, r.b));
      ProfAcc& acc = s->prof_acc[s->prof_names[r.name_id]];
      acc.launches += r.kernels;
      acc.ms += t;
      acc.flops += r.flops;
      acc.bytes += r.bytes;
    }
  }
  s->kernels_launched += n;
  FO_CUDA(cudaGetLastError());
  FO_CUDA(cudaEventRecord(s->slot_free[slot], s->cs));
  FO_CUDA(cudaEventRecord(s->step_done[s->steps_done % fo_server::kStepEvents], s->cs));
  s->slot_consumed[slot] = 1;
  s->steps_done++;
  s->last_launches = n;
  return FO_OK;
}

int fo_read_losses(fo_server* s, float* host_out, int64_t first_step, int64_t n) {
  if (!s || !host_out || first_step < 0 || n < 0 || first_step + n > s->steps_done ||
      s->steps_done - first_step > s->kLossRing)
    return set_err(FO_ERR_ARG, "loss range");
  if (n == 0) return FO_OK;
  // The event slot of the last step read holds that step or a later one:
  // either way the losses asked for are written once it has completed.
  FO_CUDA(cudaEventSynchronize(s->step_done[(first_step + n - 1) % fo_server::kStepEvents]));
  for (int64_t i = 0; i < n; ++i) {
    int64_t idx = (first_step + i) & (s->kLossRing - 1);
    FO_CUDA(cudaMemcpy(host_out + i, s->losses + idx, 4, cudaMemcpyDeviceToHost));
  }
  return FO_OK;
}

int fo_aggregate(fo_server* s, float* global, const float* local, int64_t n, int device_id,
                 int32_t version, int32_t* new_version) {
  if (!s || !global || !local || n < 0) return set_err(FO_ERR_ARG, "null argument");
  if (device_id < 0 || device_id >= s->cfg.num_devices) return set_err(FO_ERR_ARG, "bad device id");
  if (version < 0 || version > s->t) return set_err(FO_ERR_ARG, "model version out of range");
  if (int64_t(s->t) - version > s->cfg.max_delay) {
    if (new_version) *new_version = s->t;
    return FO_STALE;
  }
  float alpha = 1.0f / float(s->t - version + 1);
  cudaPointerAttributes pa{};
  FO_CUDA(cudaPointerGetAttributes(&pa, local));
  int stage_buf = -1;
  if (n > 0 && pa.type != cudaMemoryTypeDevice && pa.type != cudaMemoryTypeManaged) {
    // a host-resident local model: copied to a device buffer first
    if (n > s->agg_stage_n) {
      FO_CUDA(cudaStreamSynchronize(s->cs));
      for (int b = 0; b < 2; ++b) {
        if (s->agg_stage[b]) {
          cudaFree(s->agg_stage[b]);
          s->device_bytes -= s->agg_stage_n * 4;
          s->agg_stage[b] = nullptr;
        }
        if (cudaMalloc(&s->agg_stage[b], size_t(n) * 4) != cudaSuccess) {
          cudaGetLastError();
          s->agg_stage_n = 0;
          return set_err(FO_ERR_OOM, "aggregation staging");
        }
        s->device_bytes += n * 4;
        if (!s->agg_landed[b]) {
          FO_CUDA(cudaEventCreateWithFlags(&s->agg_landed[b], cudaEventDisableTiming));
          FO_CUDA(cudaEventCreateWithFlags(&s->agg_read[b], cudaEventDisableTiming));
        }
      }
      s->agg_stage_n = n;
    }
    stage_buf = int(s->agg_next++ & 1);
    float* dst = s->agg_stage[stage_buf];
    FO_CUDA(cudaStreamWaitEvent(s->hs, s->agg_read[stage_buf], 0));   // the aggregation that last read it
    FO_CUDA(cudaMemcpyAsync(dst, local, size_t(n) * 4, cudaMemcpyHostToDevice, s->hs));
    FO_CUDA(cudaEventRecord(s->agg_landed[stage_buf], s->hs));
    FO_CUDA(cudaStreamWaitEvent(s->as, s->agg_landed[stage_buf], 0));
    FO_CUDA(cudaEventSynchronize(s->agg_landed[stage_buf]));   // the caller may reuse `local`
    local = dst;
  }
  const int nk = fo::axpby_kernels(global, local, n);
  if (s->profiling) {
    ProfRec r{prof_id(s, "fedasync_axpby"), pool_event(s), pool_event(s), nk, 0.0, 12.0 * double(n)};
    cudaEventRecord(r.a, s->as);
    fo::axpby(global, local, n, alpha, s->as);
    cudaEventRecord(r.b, s->as);
    s->prof.push_back(r);
  } else {
    fo::axpby(global, local, n, alpha, s->as);
  }
  s->kernels_launched += nk;
  FO_CUDA(cudaGetLastError());
  if (stage_buf >= 0) FO_CUDA(cudaEventRecord(s->agg_read[stage_buf], s->as));
  s->t += 1;
  if (new_version) *new_version = s->t;
  return FO_OK;
}

int fo_get_counters(const fo_server* s, uint64_t* c) {
  if (!s || !c) return set_err(FO_ERR_ARG, "null argument");
  const auto& v = s->sched->counters();
  for (size_t i = 0; i < v.size(); ++i) c[i] = v[i];
  return FO_OK;
}
int fo_get_sender_status(const fo_server* s, uint8_t* on) {
  if (!s || !on) return set_err(FO_ERR_ARG, "null argument");
  const auto& v = s->sched->sender_on();
  for (size_t i = 0; i < v.size(); ++i) on[i] = v[i];
  return FO_OK;
}
int fo_get_version(const fo_server* s, int32_t* t, int32_t* round) {
  if (!s) return set_err(FO_ERR_ARG, "null server");
  if (t) *t = s->t;
  if (round) *round = s->t / s->cfg.num_devices;
  return FO_OK;
}
int fo_set_device_active(fo_server* s, int device_id, int active) {
  if (!s) return set_err(FO_ERR_ARG, "null server");
  return s->sched->set_active(device_id, active) == 0 ? FO_OK : set_err(FO_ERR_ARG, "bad device id");
}
int64_t fo_server_activation_bytes(const fo_server* s) {
  if (!s) return -1;
  return int64_t(s->cfg.omega) * (s->slot_stride + 2 * int64_t(s->cfg.batch) * 4);
}
int fo_server_synchronize(fo_server* s) {
  if (!s) return set_err(FO_ERR_ARG, "null server");
  FO_CUDA(cudaStreamSynchronize(s->hs));
  FO_CUDA(cudaStreamSynchronize(s->xs));
  FO_CUDA(cudaStreamSynchronize(s->cs));
  FO_CUDA(cudaStreamSynchronize(s->as));
  return FO_OK;
}
void* fo_server_stream(const fo_server* s) { return s ? (void*)s->cs : nullptr; }
void* fo_server_agg_stream(const fo_server* s) { return s ? (void*)s->as : nullptr; }
int fo_server_join_aggregations(fo_server* s) {
  if (!s) return set_err(FO_ERR_ARG, "null server");
  FO_CUDA(cudaEventRecord(s->agg_ev, s->as));
  FO_CUDA(cudaStreamWaitEvent(s->cs, s->agg_ev, 0));
  return FO_OK;
}
int fo_server_last_step_launches(const fo_server* s) { return s ? s->last_launches : -1; }

int fo_server_profile(fo_server* s, int enable) {
  if (!s) return set_err(FO_ERR_ARG, "null server");
  s->profiling = enable != 0;
  return FO_OK;
}

int fo_server_kernel_times(fo_server* s, const char** names, int64_t* launches, double* ms,
                           double* flops, double* bytes, int cap, int* n_out) {
  if (!s || !n_out) return set_err(FO_ERR_ARG, "null argument");
  FO_CUDA(cudaStreamSynchronize(s->cs));
  for (auto& r : s->prof) {
    float t = 0.f;
    cudaEventElapsedTime(&t, r.a, r.b);
    ProfAcc& acc = s->prof_acc[s->prof_names[r.name_id]];
    acc.launches += r.kernels;
    acc.ms += t;
    acc.flops += r.flops;
    acc.bytes += r.bytes;
    s->ev_pool.push_back(r.a);
    s->ev_pool.push_back(r.b);
  }
  s->prof.clear();
  int n = 0;
  for (auto& kv : s->prof_acc) {
    if (n < cap) {
      if (names) names[n] = kv.first;
      if (launches) launches[n] = kv.second.launches;
      if (ms) ms[n] = kv.second.ms;
      if (flops) flops[n] = kv.second.flops;
      if (bytes) bytes[n] = kv.second.bytes;
    }
    ++n;
  }
  *n_out = n;
  return FO_OK;
}

int fo_server_profile_reset(fo_server* s) {
  if (!s) return set_err(FO_ERR_ARG, "null server");
  FO_CUDA(cudaStreamSynchronize(s->cs));
  for (auto& r : s->prof) {
    s->ev_pool.push_back(r.a);
    s->ev_pool.push_back(r.b);
  }
  s->prof.clear();
  s->prof_acc.clear();
  return FO_OK;
}

int64_t fo_server_kernels_launched(const fo_server* s) { return s ? s->kernels_launched : -1; }

int64_t fo_server_device_bytes(const fo_server* s) { return s ? s->device_bytes : -1; }

int fo_server_error(fo_server* s) {
  if (!s) return set_err(FO_ERR_ARG, "null server");
  int* w = fo::tc_error_word(s->tc);
  if (!w) return FO_OK;
  int h = 0;
  FO_CUDA(cudaStreamSynchronize(s->cs));
  FO_CUDA(cudaMemcpy(&h, w, sizeof(int), cudaMemcpyDeviceToHost));
  return h ? set_err(FO_ERR_TIMEOUT, "a tensor-core kernel timed out waiting (code " + std::to_string(h) + ")") : FO_OK;
}

int fo_column_sums(const void* x, int dtype, int64_t rows, int cols, float* out, void* stream) {
  if (!x || !out || rows < 1 || cols < 1 || (dtype != FO_DTYPE_F32 && dtype != FO_DTYPE_BF16))
    return set_err(FO_ERR_ARG, "bad column-sum arguments");
  if (rows > fo::kColsumMaxRows)
    return set_err(FO_ERR_ARG, "fo_column_sums: " + std::to_string(rows) + " rows exceed " +
                                   std::to_string(fo::kColsumMaxRows) + " (65,535 chunks of 128 rows)");
  cudaStream_t st = (cudaStream_t)stream;
  float* ws = nullptr;
  FO_CUDA(cudaMallocAsync((void**)&ws, fo::colsum_partial_floats(rows, cols) * sizeof(float), st));
  fo::colsum(x, nullptr, rows, cols, dtype == FO_DTYPE_F32 ? fo::kF32 : fo::kBF16, ws, out, st);
  cudaError_t e = cudaGetLastError();
  cudaFreeAsync(ws, st);
  if (e != cudaSuccess) return set_err(FO_ERR_CUDA, cudaGetErrorString(e));
  return FO_OK;
}

int fo_axpby_async(float* global, const float* local, int64_t n, float alpha, void* stream) {
  if (!global || !local || n < 0 || !(alpha > 0.f) || alpha > 1.f) return set_err(FO_ERR_ARG, "bad argument");
  fo::axpby(global, local, n, alpha, (cudaStream_t)stream);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return set_err(FO_ERR_CUDA, cudaGetErrorString(e));
  return FO_OK;
}

// ------------------------------------------------------ host-only scheduler
struct fo_sched {
  fo::TaskScheduler* s;
};

int fo_sched_create(int K, int omega, int depth, int policy, fo_sched** out) {
  if (!out || K <= 0 || K > FO_MAX_DEVICES || omega <= 0 || omega > FO_MAX_OMEGA || depth <= 0 ||
      (policy != FO_SCHED_COUNTER && policy != FO_SCHED_FIFO))
    return set_err(FO_ERR_ARG, "bad scheduler configuration");
  *out = nullptr;
  fo::TaskScheduler* t = nullptr;
  try {
    t = new fo::TaskScheduler(K, omega, depth, policy);
    *out = new fo_sched{t};
  } catch (const std::bad_alloc&) {
    delete t;
    return set_err(FO_ERR_OOM, "host allocation");
  }
  return FO_OK;
}
int fo_sched_destroy(fo_sched* s) {
  if (s) {
    delete s->s;
    delete s;
  }
  return FO_OK;
}
int fo_sched_put(fo_sched* s, int k, int32_t* slot, int* sender_on) {
  if (!s || !slot) return set_err(FO_ERR_ARG, "null argument");
  *slot = -1;
  if (k < 0 || k >= s->s->K()) return set_err(FO_ERR_ARG, "bad device id");
  int rc = s->s->put(k, slot);
  if (sender_on) *sender_on = s->s->sender_on()[k];
  return rc == -1 ? set_err(FO_ERR_ARG, "device has left") : (rc == 2 ? FO_FULL : FO_OK);
}
int fo_sched_get(fo_sched* s, int* k, int32_t* slot) {
  if (!s || !k || !slot) return set_err(FO_ERR_ARG, "null argument");
  *k = -1;
  *slot = -1;
  return s->s->get(k, slot) == 0 ? FO_OK : FO_EMPTY;
}
int fo_sched_set_active(fo_sched* s, int k, int active) {
  if (!s) return set_err(FO_ERR_ARG, "null argument");
  return s->s->set_active(k, active) == 0 ? FO_OK : set_err(FO_ERR_ARG, "bad device id");
}
int fo_sched_counters(const fo_sched* s, uint64_t* c) {
  if (!s || !c) return set_err(FO_ERR_ARG, "null argument");
  const auto& v = s->s->counters();
  for (size_t i = 0; i < v.size(); ++i) c[i] = v[i];
  return FO_OK;
}
int fo_sched_sender_status(const fo_sched* s, uint8_t* on) {
  if (!s || !on) return set_err(FO_ERR_ARG, "null argument");
  const auto& v = s->s->sender_on();
  for (size_t i = 0; i < v.size(); ++i) on[i] = v[i];
  return FO_OK;
}
int fo_sched_queued(const fo_sched* s, int k) {
  if (!s) return -1;
  if (k < 0) return s->s->queued_total();
  if (k >= s->s->K()) return -1;
  return s->s->queued(k);
}

}  // extern "C"
