// Internal state of a FedOptima server (shared by the plan builder and the
// tensor-core planner).
#pragma once
#include "fo_common.cuh"
#include "fo_kernels.h"
#include "fo_sched.hpp"
#include "../../include/fedoptima.h"

#include <functional>
#include <map>
#include <string>
#include <vector>

namespace fo {
struct TcContext;
struct AttnTcPlan;
}

struct ParamSeg {
  int op;
  int64_t off;   // offset in the padded device vector
  int64_t flat;  // offset in the caller's flat vector
  int64_t n;
};

struct Tensor {
  int N = 0, H = 0, W = 0, C = 0;
  int dt = fo::kF32;
  void* act = nullptr;
  void* grad = nullptr;
  int root = -1;        // tensor whose buffers this one aliases (flatten), else itself
  int consumers = 0;
  int64_t rows() const { return int64_t(N) * H * W; }
  int64_t numel() const { return rows() * C; }
  size_t bytes() const { return size_t(numel()) * (dt == fo::kF32 ? 4 : 2); }
  // The uploaded batch (tensor 0) or a view of it (a flatten of the input):
  // its data is the current batch slot, and it has no gradient.
  bool is_input() const { return root == 0; }
};

struct Launch {
  const char* name;
  std::function<void(cudaStream_t)> fn;
  int kernels;     // kernel launches this entry makes
  double flops;    // algorithmic FLOPs
  double bytes;    // algorithmic HBM bytes
  int lane = 0;    // 1: a weight gradient, which the step graph runs on the side stream;
                   // 2: an early weight update, on the optimizer stream
  bool join = false;   // the step graph joins the side stream before this entry
};

struct ProfRec {
  int name_id;
  cudaEvent_t a, b;
  int kernels;
  double flops, bytes;
};

struct ProfAcc {
  int64_t launches = 0;
  double ms = 0, flops = 0, bytes = 0;
};

struct fo_server {
  fo_server_cfg cfg{};
  fo_optimizer opt{};
  std::vector<fo_op> ops;
  fo::TaskScheduler* sched = nullptr;
  cudaStream_t cs = nullptr, xs = nullptr;
  // Uploads: the host-to-device copy of the caller's buffers runs on `hs`
  // and never waits for compute.  An upload whose slot a queued step still
  // reads lands in a device staging buffer first and moves into the slot on
  // `xs` once that step has finished, so the caller returns as soon as its
  // own copy is done instead of waiting for the step.
  cudaStream_t hs = nullptr;
  static constexpr int kStage = 3;
  char* stage_buf = nullptr;
  int64_t stage_stride = 0;
  std::vector<cudaEvent_t> stage_landed, stage_free;
  int64_t stage_next = 0;
  // Side stream of the step graph: the weight gradients run on it, forked
  // from the compute stream after their output gradient is ready and joined
  // before the optimizer, so they fill the SMs the input-gradient chain
  // leaves idle.  Events are capture-time fork / join points.
  cudaStream_t side = nullptr;
  cudaEvent_t fork_ev = nullptr, join_ev = nullptr;
  // Optimizer stream: the update of a weight tensor, forked once both its
  // gradient (side stream) and its layer's input gradient (compute stream)
  // are done, so the HBM-bound update overlaps the GEMMs that follow.
  cudaStream_t opt_st = nullptr;
  cudaEvent_t fork2_ev = nullptr, join2_ev = nullptr;
  // Aggregation stream: FedAsync updates of device models touch no data of
  // the training step, so they run here and overlap the steps; agg_ev lets
  // the compute stream join them (fo_server_join_aggregations).
  cudaStream_t as = nullptr;
  cudaEvent_t agg_ev = nullptr;
  bool use_side = true;
  int dt = fo::kF32;

  int64_t n_params = 0, n_padded = 0;
  std::vector<ParamSeg> segs;
  std::vector<std::vector<int>> op_segs;  // per op: indices into segs
  float *theta = nullptr, *mom = nullptr, *grad = nullptr;
  fo::bf16* shadow = nullptr;

  int64_t slot_act_bytes = 0, slot_stride = 0;
  char* slab = nullptr;
  int32_t* slot_labels = nullptr;
  int32_t* slot_lengths = nullptr;
  std::vector<cudaEvent_t> slot_ready, slot_free;
  std::vector<char> slot_consumed;

  std::vector<Tensor> T;
  float* colsum_scratch = nullptr;
  std::vector<float*> ln_mean, ln_rstd, attn_probs;
  float* simt_scratch = nullptr;   // K-split partials of the CUDA-core weight gradient

  const void* cur_in = nullptr;
  const int32_t* cur_labels = nullptr;
  const int32_t* cur_len = nullptr;
  float* losses = nullptr;
  float* row_loss = nullptr;
  int64_t* d_step = nullptr;   // device copy of steps_done (indexes the loss ring)
  bool use_graphs = true;
  std::vector<cudaGraphExec_t> graphs, prof_graphs;  // per batch slot
  std::vector<std::vector<struct ProfRec>> prof_events;
  int64_t steps_done = 0;
  static constexpr int64_t kLossRing = int64_t(1) << 20;
  // Completion events of the most recent steps (step i records slot i % 64),
  // so that reading a step's loss waits for that step only.
  static constexpr int kStepEvents = 64;
  std::vector<cudaEvent_t> step_done;
  // Device copies of host-resident local models for fo_aggregate: two
  // buffers, so that the upload of one model overlaps the aggregation of the
  // previous one (landed: copy done; read: the aggregation that used it).
  float* agg_stage[2] = {nullptr, nullptr};
  int64_t agg_stage_n = 0;
  cudaEvent_t agg_landed[2] = {nullptr, nullptr}, agg_read[2] = {nullptr, nullptr};
  int64_t agg_next = 0;

  std::vector<Launch> plan;
  int last_launches = 0;

  int32_t t = 0;

  bool profiling = false;
  std::vector<ProfRec> prof;
  std::vector<cudaEvent_t> ev_pool;
  std::vector<const char*> prof_names;
  std::map<const char*, ProfAcc> prof_acc;
  int64_t kernels_launched = 0;
  int64_t device_bytes = 0;

  std::vector<void*> allocs;
  fo::TcContext* tc = nullptr;
  std::vector<fo::AttnTcPlan*> attn_tc;   // per op: tensor-core attention plan, or null

  void* alloc(size_t bytes) {
    void* p = nullptr;
    if (bytes == 0) bytes = 256;
    if (cudaMalloc(&p, bytes) != cudaSuccess) return nullptr;
    allocs.push_back(p);
    device_bytes += int64_t(bytes);
    return p;
  }
  int op_of_tensor(int tid) const { return tid - 1; }
};

