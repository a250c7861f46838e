// Planner of the tensor-core GEMM / implicit-GEMM convolution kernels
// (tc_gemm_kernels.cuh): tensor maps, tile width and K split from a cost
// model, epilogue variant, split-K workspaces and launches.
#include "fo_server_impl.h"
#include "fo_tc.h"
#include "tc_gemm_kernels.cuh"

#include <cuda.h>
#include <algorithm>
#include <cstring>
#include <map>
#include <vector>

namespace fo {

using namespace tcg;

namespace {

// The epilogue variant a plan's parameters ask for.
int epi_of(const TcParams& p) {
  return (p.out_f32 ? E_F32 : 0) | (p.relu ? E_RELU : 0) | (p.mask ? E_MASK : 0) | (p.acc ? E_ACC : 0) |
         (p.pool_out ? E_POOL : 0) | (p.tma_out ? E_TMA : 0) | (p.gelu_out ? E_GELU : 0);
}

KernelFn pick_kernel(int kind, int bn, bool cluster, int epi, size_t* smem) {
  switch (kind) {
    case LIN_FWD:
    case CONV_FPROP:
      return pick_fwd(kind, bn, cluster, epi, smem);
    case LIN_DGRAD:
    case CONV_DGRAD:
      return pick_dgrad(kind, bn, cluster, epi, smem);
    case LIN_WGRAD:
    case CONV_WGRAD:
      return pick_wgrad(kind, bn, cluster, epi, smem);
  }
  return nullptr;
}

// ------------------------------------------------------------ tensor maps
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// bf16 tensor map, dims innermost first, strides in bytes of dims 1.. .
// elem (may be null): traversal step per dimension (the box then spans
// box[i] elements and loads box[i] / elem[i] of them).
bool make_map(CUtensorMap* m, const void* base, int rank, const uint64_t* dims, const uint64_t* strides,
              const uint32_t* box, const uint32_t* elem = nullptr,
              CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t d[5], st[4];
  cuuint32_t b[5], es[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    b[i] = box[i];
    es[i] = elem ? elem[i] : 1;
    if (i + 1 < rank) st[i] = strides[i];
  }
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), d, st, b, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 2-D [rows][cols] row-major bf16, box (64 cols, box_rows).
bool map_2d(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int box_rows) {
  uint64_t dims[2] = {uint64_t(cols), uint64_t(rows)};
  uint64_t strides[1] = {uint64_t(cols) * 2};
  uint32_t box[2] = {64, uint32_t(box_rows)};
  return make_map(m, base, 2, dims, strides, box);
}

// The output of an E_TMA GEMM: bf16 [rows][cols] with row pitch ld, box 32
// columns x 32 rows, 64-byte swizzle (the epilogue's staging layout).
bool map_out(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int64_t ld) {
  if (ld % 8 || cols > ld || (reinterpret_cast<uintptr_t>(base) & 15)) return false;
  uint64_t dims[2] = {uint64_t(cols), uint64_t(rows)};
  uint64_t strides[1] = {uint64_t(ld) * 2};
  uint32_t box[2] = {32, 32};
  return make_map(m, base, 2, dims, strides, box, nullptr, CU_TENSOR_MAP_SWIZZLE_64B);
}

// 4-D NHWC window map over an N x H x W x C tensor that loads, per box,
// 64 channels x ow columns x rows x imgs, stepping `stride` pixels in H and W
// (the box spans ow*stride columns and rows*stride rows of the tensor).
// [rows][cols] seen as {64, rows, cols / 64} (cols % 64 == 0): a box of
// `chunks` 64-column chunks x box_rows rows lands chunk after chunk, each
// box_rows x 128 bytes, the layout of an MN-major operand.
bool map_chunked(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int box_rows, int chunks) {
  if (cols % 64) return false;
  uint64_t dims[3] = {64, uint64_t(rows), uint64_t(cols / 64)};
  uint64_t strides[2] = {uint64_t(cols) * 2, 128};
  uint32_t box[3] = {64, uint32_t(box_rows), uint32_t(chunks)};
  return make_map(m, base, 3, dims, strides, box);
}
// The windowed NHWC tensor of map_window with its channels split the same
// way: {64, W, H, N, C / 64}, `chunks` channel chunks per box (C % 64 == 0).
bool map_window_chunked(CUtensorMap* m, const void* base, int N, int H, int W, int C, int ow, int rows, int imgs,
                        int stride, int chunks) {
  if (C % 64) return false;
  uint64_t dims[5] = {64, uint64_t(W), uint64_t(H), uint64_t(N), uint64_t(C / 64)};
  uint64_t strides[4] = {uint64_t(C) * 2, uint64_t(W) * C * 2, uint64_t(H) * W * C * 2, 128};
  uint32_t box[5] = {64, uint32_t(ow * stride), uint32_t(rows * stride), uint32_t(imgs), uint32_t(chunks)};
  uint32_t elem[5] = {1, uint32_t(stride), uint32_t(stride), 1, 1};
  return make_map(m, base, 5, dims, strides, box, elem);
}
bool map_window(CUtensorMap* m, const void* base, int N, int H, int W, int C, int ow, int rows, int imgs,
                int stride = 1) {
  uint64_t dims[4] = {uint64_t(C), uint64_t(W), uint64_t(H), uint64_t(N)};
  uint64_t strides[3] = {uint64_t(C) * 2, uint64_t(W) * C * 2, uint64_t(H) * W * C * 2};
  uint32_t box[4] = {64, uint32_t(ow * stride), uint32_t(rows * stride), uint32_t(imgs)};
  uint32_t elem[4] = {1, uint32_t(stride), uint32_t(stride), 1};
  return make_map(m, base, 4, dims, strides, box, elem);
}

}  // namespace

// ------------------------------------------------------------------ plans
struct TcGemm {
  // Every field starts at zero / null (the kernel parameters included);
  // only the window stride defaults to 1.
  TcGemm() : p{} { p.stride = 1; }
  const char* name = nullptr;
  int kind = 0, bn = 0, splits = 1;
  double flops = 0;
  TcParams p;
  KernelFn fn = nullptr;
  size_t smem = 0;
  dim3 grid;
  int lane = 0;           // stream lane (split-K workspace per lane)
  bool input_A = false;   // operand fed by the uploaded batch (tensor 0 or a view of it)
  bool input_B = false;
  bool input_acc = false; // the epilogue's addend is the uploaded batch
  std::vector<CUtensorMap> slot_maps;  // per slot map of that operand
  TcContext* ctx = nullptr;
};

struct TcContext {
  std::vector<TcGemm*> gemms;
  std::map<int, int> cluster_fit;   // active_clusters() cache
  int num_sms = 148;
  int slot = 0;
  int* err = nullptr;
  fo_server* s = nullptr;
  float* ws[2] = {nullptr, nullptr};   // split-K workspace per stream lane (a lane's GEMMs run in order)
};

namespace {

bool window_ok(int N, int H, int W, int rows_needed, int* rows, int* imgs) {
  // A box of `rows_needed` pixels made of whole image rows (and whole images
  // when it spans several).
  if (W > 256 || rows_needed % W) return false;
  int r = rows_needed / W;
  if (r <= H) {
    if (H % r) return false;
    *rows = r;
    *imgs = 1;
  } else {
    if (r % H) return false;
    *rows = H;
    *imgs = r / H;
    if (*imgs > 256) return false;
  }
  (void)N;
  return true;
}


// Split-K clusters of S CTAs of kernel (kind, bn) that fit on the GPU at
// once (GPC packing), from the occupancy calculator; cached per context.
int active_clusters(TcContext* c, int kind, int bn, int S, int epi) {
  const int key = ((kind * 512 + bn) * 16 + S) * 16 + epi;
  auto it = c->cluster_fit.find(key);
  if (it != c->cluster_fit.end()) return it->second;
  size_t smem = 0;
  KernelFn fn = pick_kernel(kind, bn, true, epi, &smem);
  int n = 0;
  if (fn && cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1, 1, S);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 1;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = S;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();
  if (n <= 0)   // conservative fallback
    n = c->num_sms / (2 * S) > 0 ? c->num_sms / (2 * S) : 1;
  c->cluster_fit[key] = n;
  return n;
}

// Tile width and K split from a cost model in microseconds,
// fitted to GB300 timelines of these kernels:
//  * a k-block stage costs at least ~0.37 us: each stage is one round of
//    mbarrier waits (full on the MMA side, empty on the TMA side), whose
//    dependent latency is a few hundred cycles on each side;
//  * the TMA fills one SM's shared memory at ~128 GB/s, which bounds stages
//    of 256-wide tiles (48 KB);
//  * a stage issues four 128 x BN x 16 MMAs, and each takes ~190 cycles
//    whatever BN <= 256 (measured: 128- and 256-wide weight-gradient stages
//    both ~0.38-0.40 us once all chunks of an operand come in one TMA box),
//    so 256-wide tiles run at the measured dense bf16 rate (about 3/4 of
//    the nominal one) and 128-wide ones at half of it: the floor above;
//  * a CTA pays a start-up ramp and the epilogue of its last tile (earlier
//    epilogues overlap the next tile's MMAs), a K-split cluster pays the
//    exchange of its partial tiles through the L2 workspace and their
//    reduction, and clusters run in waves of what the occupancy calculator
//    fits at once.
// Candidate widths divide `ndiv` (N, or the channels of one tap for the
// weight gradient, whose N index runs over taps x channels); a weight-gradient
// tile may instead span two whole taps, one TMA box per tap.
void choose_tiles(TcContext* c, TcGemm* g, int M, int N, int KB, int ndiv) {
  const bool win_a = g->kind == CONV_FPROP || g->kind == CONV_DGRAD;
  const bool win_b = g->kind == CONV_WGRAD;
  double best = 1e30;
  int best_bn = 0, best_s = 1;
  for (int bn : {256, 128, 64}) {
    // window kinds tile whole taps; the plain GEMMs take a ragged last tile,
    // and so does a weight gradient whose tiles span (at most two) taps
    if (win_a && (ndiv % bn || N % bn)) continue;
    if (win_b && ndiv % bn && (bn % ndiv || bn > 2 * ndiv)) continue;
    const int n_tiles = (N + bn - 1) / bn, m_tiles = (M + BM - 1) / BM, tiles = n_tiles * m_tiles;
    const double stage_kb = (BM + bn) * BK * 2 / 1024.0;
    const double epi = bn == 256 ? 4.2 : (bn == 128 ? 2.2 : 1.5);
    double t_kb = std::max(0.37, stage_kb / 128.0);
    if (win_b) t_kb = std::max(t_kb, 0.39);
    for (int sp = 1; sp <= 8; ++sp) {
      if (sp > 1 && KB / sp < 4) break;
      // an owner's receive slices (16 KB per other rank and owned chunk) live in the pipeline buffers
      if (sp > 1 && size_t(sp - 1) * ((bn / 32 + sp - 1) / sp) * 16384 > pipeline_bytes(bn)) continue;
      const int kper = (KB + sp - 1) / sp;
      const int splits = (KB + kper - 1) / kper;
      if (splits != sp) continue;
      double cost;
      if (splits == 1) {
        const int units = std::min(tiles, c->num_sms);
        const int per_unit = (tiles + units - 1) / units;
        const double main = kper * t_kb;
        cost = 1.7 + per_unit * main + epi + (per_unit - 1) * std::max(0.0, epi - main);
      } else {
        const int fit = active_clusters(c, g->kind, bn, splits, epi_of(g->p));
        const int waves = (tiles + fit - 1) / fit;
        cost = waves * (1.0 + kper * t_kb + 3.0 + 2.5 * bn / 128.0);
      }
      if (cost < best - 1e-9) {
        best = cost;
        best_bn = bn;
        best_s = splits;
      }
    }
  }
  g->bn = best_bn;
  g->p.KB = KB;
  g->p.kper = (KB + best_s - 1) / best_s;
  g->splits = best_s;
}

TcGemm* finish(TcContext* c, TcGemm* g, int M, int N, double K) {
  if (g->p.acc && !g->p.accsrc && !g->input_acc) g->p.accsrc = static_cast<const bf16*>(g->p.out);
  g->p.M = M;
  g->p.N = N;
  g->flops = 2.0 * M * N * K;
  g->p.err = c->err;
  // An unsplit plan with a plain bf16 output stores it by TMA from an
  // accumulator that starts from the bias (E_TMA).
  if (g->splits == 1 && !(epi_of(g->p) & (E_F32 | E_POOL)) && !g->p.ostride && !getenv("FO_NO_TMA_STORE") &&
      map_out(&g->p.tmO, g->p.out, M, N, g->p.ldo))
    g->p.tma_out = 1;
  // The GELU epilogue exists only in that form (a split plan runs the GELU
  // as its own kernel: the caller plans again without it).
  if (g->p.gelu_out && (!g->p.tma_out || !map_out(&g->p.tmG, g->p.gelu_out, M, N, g->p.ldo))) {
    delete g;
    return nullptr;
  }
  g->fn = pick_kernel(g->kind, g->bn, g->splits > 1, epi_of(g->p), &g->smem);
  if (!g->fn) {
    delete g;
    return nullptr;
  }
  if (cudaFuncSetAttribute(g->fn, cudaFuncAttributeMaxDynamicSharedMemorySize, int(g->smem)) != cudaSuccess) {
    delete g;
    return nullptr;
  }
  const int n_tiles = (N + g->bn - 1) / g->bn;
  if (g->splits > 1) {
    g->grid = dim3(n_tiles, (M + BM - 1) / BM, g->splits);
  } else {
    const int tiles = n_tiles * ((M + BM - 1) / BM);
    g->grid = dim3(std::min(tiles, c->num_sms), 1, 1);
  }
  if (getenv("FO_DEBUG_PLAN"))
    fprintf(stderr, "[plan] %-16s M=%d N=%d KB=%d BN=%d splits=%d grid=(%u,%u,%u) chunked=%d%d\n", g->name, M, N,
            g->p.KB, g->bn, g->splits, g->grid.x, g->grid.y, g->grid.z, g->p.chunk_a, g->p.chunk_b);
  g->ctx = c;
  c->gemms.push_back(g);
  return g;
}

bool bf16_server(const fo_server* s) { return s->dt == kBF16; }

}  // namespace

int tc_create(TcContext** out, fo_server* s) {
  TcContext* c = new TcContext();
  c->s = s;
  int dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, dev);
  c->err = (int*)s->alloc(sizeof(int) * 4);
  if (!c->err) {
    delete c;
    return FO_ERR_OOM;
  }
  cudaMemset(c->err, 0, sizeof(int) * 4);
  *out = c;
  return FO_OK;
}

void tc_destroy(TcContext* c) {
  if (!c) return;
  for (TcGemm* g : c->gemms) delete g;
  delete c;
}

void tc_set_input(TcContext* c, int slot) {
  if (c) c->slot = slot;
}

bool tc_encode_2d(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int box_rows) {
  return map_2d(m, base, rows, cols, box_rows);
}

int* tc_error_word(TcContext* c) { return c ? c->err : nullptr; }

void tc_set_lane(TcGemm* g, int lane) {
  if (g) g->lane = lane ? 1 : 0;
}

// Allocate the split-K workspaces once every plan is known: the GEMMs of one
// stream lane run one after another, so they share that lane's workspace.
int tc_finalize(TcContext* c) {
  if (!c) return FO_OK;
  size_t need[2] = {0, 0};
  for (TcGemm* g : c->gemms)
    if (g->splits > 1)
      need[g->lane] = std::max(need[g->lane], size_t(g->grid.x) * g->grid.y * g->splits * BM * g->bn);
  for (int l = 0; l < 2; ++l) {
    if (!need[l]) continue;
    c->ws[l] = static_cast<float*>(c->s->alloc(need[l] * sizeof(float)));
    if (!c->ws[l]) return FO_ERR_OOM;
  }
  for (TcGemm* g : c->gemms)
    if (g->splits > 1) g->p.ws = c->ws[g->lane];
  return FO_OK;
}

static const void* tensor_act(fo_server* s, int tid) { return s->T[tid].act; }

// Linear layers and 1x1 stride-1 convolutions are one plain GEMM over the
// rows of an NHWC tensor.  Channel counts need only be multiples of 8 (rows
// of 16 bytes for the tensor maps): a ragged contraction block is zero-filled
// by the TMA, and a ragged last output tile is masked in the epilogue.
static bool plain_gemm(const fo_op& op) {
  return op.kind == FO_OP_LINEAR || (op.kind == FO_OP_CONV && op.k == 1 && op.stride == 1);
}
static bool plain_gemm_ok(const fo_op& op) { return op.cin % 8 == 0 && op.cout % 8 == 0; }

bool tc_plain_ok(TcContext* c, const fo_server* s, int i) {
  if (!c || !bf16_server(s) || getenv("FO_NO_TC")) return false;
  const fo_op& op = s->ops[i];
  return plain_gemm(op) && plain_gemm_ok(op) && s->T[i + 1].dt == kBF16;
}

static void apply_epilogue(TcGemm* g, const TcEpilogue* ex) {
  if (!ex) return;
  g->p.pool_out = static_cast<bf16*>(ex->pool_out);
  g->p.pool_code = ex->pool_code;
  g->p.gelu_out = static_cast<bf16*>(ex->gelu_out);
  if (ex->addend || ex->addend_is_input) {
    g->p.acc = 1;
    g->p.accsrc = static_cast<const bf16*>(ex->addend);
    g->input_acc = ex->addend_is_input;
  }
}

TcGemm* tc_plan_forward(TcContext* c, fo_server* s, int i, void* out, bool relu, const TcEpilogue* ex) {
  if (!c || !bf16_server(s) || getenv("FO_NO_TC")) return nullptr;
  const fo_op& op = s->ops[i];
  const Tensor& a = s->T[op.in0];
  const Tensor& o = s->T[i + 1];
  if (o.dt != kBF16) return nullptr;  // fp32 logits: CUDA-core path
  if (ex && (ex->addend || ex->addend_is_input) && (relu || !plain_gemm(op))) return nullptr;
  if (ex && ex->gelu_out && (relu || !plain_gemm(op) || ex->pool_out || ex->addend || ex->addend_is_input))
    return nullptr;
  if (ex && ex->pool_out) {   // whole 2 x 2 windows inside each warp's 32 rows
    const bool w_ok = o.W == 2 || o.W == 4 || o.W == 8 || o.W == 16;
    if (!relu || !w_ok || o.H % 2 || o.C % 8 || o.rows() % BM) return nullptr;
  }
  TcGemm* g = new TcGemm();
  g->p.out = out;
  g->p.ldo = o.C;
  g->p.relu = relu ? 1 : 0;
  g->p.pool_w = o.W;
  apply_epilogue(g, ex);
  g->p.bias = op.bias ? s->theta + s->segs[s->op_segs[i][1]].off : nullptr;
  const bf16* w = s->shadow + s->segs[s->op_segs[i][0]].off;
  if (plain_gemm(op)) {
    if (!plain_gemm_ok(op)) { delete g; return nullptr; }
    g->kind = LIN_FWD;
    g->name = op.kind == FO_OP_LINEAR ? "tc_linear_fwd" : "tc_conv1x1_fwd";
    int M = int(a.rows()), KB = (op.cin + 63) / 64;
    choose_tiles(c, g, M, op.cout, KB, op.cout);
    const int bn = g->bn;
    g->input_A = s->T[op.in0].is_input();
    if (g->input_A) {
      g->slot_maps.resize(s->cfg.omega);
      for (int sl = 0; sl < s->cfg.omega; ++sl)
        if (!map_2d(&g->slot_maps[sl], s->slab + size_t(sl) * s->slot_stride, M, op.cin, BM)) { delete g; return nullptr; }
    } else if (!map_2d(&g->p.tmA, tensor_act(s, op.in0), M, op.cin, BM)) { delete g; return nullptr; }
    if (!map_2d(&g->p.tmB, w, op.cout, op.cin, bn)) { delete g; return nullptr; }
    return finish(c, g, M, op.cout, double(op.cin));
  }
  // convolution: k in {1, 3}, stride in {1, 2}; tiles of 128 output pixels
  const int st = op.stride, Ho = o.H, Wo = o.W;
  if (op.cin % 64 || op.cout % 64 || (st == 2 && (a.H != 2 * Ho || a.W != 2 * Wo))) { delete g; return nullptr; }
  int rows, imgs;
  if (!window_ok(a.N, Ho, Wo, BM, &rows, &imgs) || (int64_t(a.N) * Ho * Wo) % BM) { delete g; return nullptr; }
  g->kind = CONV_FPROP;
  g->name = "tc_conv_fprop";
  g->p.H = Ho; g->p.W = Wo; g->p.ksz = op.k; g->p.pad = op.k / 2; g->p.taps = op.k * op.k; g->p.stride = st;
  g->p.cblocks = op.cin / 64;
  g->p.ntap_ch = op.cin;
  g->p.win_rows = rows; g->p.win_imgs = imgs;
  int M = a.N * Ho * Wo, KB = g->p.taps * g->p.cblocks;
  choose_tiles(c, g, M, op.cout, KB, op.cout);
  const int bn = g->bn;
  const int box_rows = rows, box_imgs = imgs;
  g->input_A = s->T[op.in0].is_input();
  if (g->input_A) {
    g->slot_maps.resize(s->cfg.omega);
    for (int sl = 0; sl < s->cfg.omega; ++sl)
      if (!map_window(&g->slot_maps[sl], s->slab + size_t(sl) * s->slot_stride, a.N, a.H, a.W, a.C, Wo, box_rows, box_imgs, st)) { delete g; return nullptr; }
  } else if (!map_window(&g->p.tmA, tensor_act(s, op.in0), a.N, a.H, a.W, a.C, Wo, box_rows, box_imgs, st)) { delete g; return nullptr; }
  if (!map_2d(&g->p.tmB, w, op.cout, int64_t(g->p.taps) * op.cin, bn)) { delete g; return nullptr; }
  return finish(c, g, M, op.cout, double(g->p.taps) * op.cin);
}

bool tc_plan_dgrad(TcContext* c, fo_server* s, int i, int accumulate, void* dx, const void* mask,
                   std::vector<TcGemm*>* out, bool* zero_first, const TcEpilogue* ex) {
  out->clear();
  *zero_first = false;
  if (!c || !bf16_server(s) || getenv("FO_NO_TC")) return false;
  const fo_op& op = s->ops[i];
  const Tensor& a = s->T[op.in0];
  const Tensor& o = s->T[i + 1];
  if (o.dt != kBF16) return false;
  if (ex && (!plain_gemm(op) || ex->addend_is_input || (ex->addend && accumulate))) return false;
  const bf16* w = s->shadow + s->segs[s->op_segs[i][0]].off;
  auto base = [&]() {
    TcGemm* g = new TcGemm();
    g->p.out = dx;
    g->p.ldo = a.C;
    g->p.acc = accumulate;
    g->p.mask = static_cast<const bf16*>(mask);
    return g;
  };
  if (plain_gemm(op)) {
    if (!plain_gemm_ok(op)) return false;
    TcGemm* g = base();
    apply_epilogue(g, ex);
    g->kind = LIN_DGRAD;
    g->name = op.kind == FO_OP_LINEAR ? "tc_linear_dgrad" : "tc_conv1x1_dgrad";
    int M = int(a.rows()), KB = (op.cout + 63) / 64;
    choose_tiles(c, g, M, op.cin, KB, op.cin);
    if (!map_2d(&g->p.tmA, o.grad, M, op.cout, BM) || !map_2d(&g->p.tmB, w, op.cout, op.cin, BK)) { delete g; return false; }
    CUtensorMap cb;
    if (map_chunked(&cb, w, op.cout, op.cin, BK, g->bn / 64)) { g->p.tmB = cb; g->p.chunk_b = 1; }
    if (!finish(c, g, M, op.cin, double(op.cout))) return false;
    out->push_back(g);
    return true;
  }
  // Convolution input gradient, split by output parity (py, px) for stride 2:
  // input row y = st*i + py receives output row p = i + dh from tap r when
  // st*dh = py + pad - r.  Each class is an implicit GEMM over its own taps.
  const int st = op.stride, pad = op.k / 2, Ho = o.H, Wo = o.W;
  if (op.cin % 64 || op.cout % 64 || (st == 2 && (a.H != 2 * Ho || a.W != 2 * Wo))) return false;
  int rows, imgs;
  if (!window_ok(o.N, Ho, Wo, BM, &rows, &imgs) || (int64_t(o.N) * Ho * Wo) % BM) return false;
  const int nclass = st * st;
  bool any_empty = false;
  struct Cls { int n; int rs[9], dh[9], dw[9]; } cls[4];
  for (int q = 0; q < nclass; ++q) {
    const int py = q / st, px = q % st;
    cls[q].n = 0;
    for (int r = 0; r < op.k; ++r)
      for (int sx = 0; sx < op.k; ++sx) {
        const int vh = py + pad - r, vw = px + pad - sx;
        if (vh % st || vw % st) continue;
        int& n = cls[q].n;
        cls[q].rs[n] = r * op.k + sx;
        cls[q].dh[n] = vh / st;
        cls[q].dw[n] = vw / st;
        ++n;
      }
    if (cls[q].n == 0) any_empty = true;
  }
  const int eff_acc = any_empty && !accumulate ? 1 : accumulate;
  *zero_first = any_empty && !accumulate;
  for (int q = 0; q < nclass; ++q) {
    if (cls[q].n == 0) continue;
    TcGemm* g = base();
    g->p.acc = eff_acc;
    g->kind = CONV_DGRAD;
    g->name = "tc_conv_dgrad";
    g->p.H = Ho; g->p.W = Wo; g->p.ksz = op.k; g->p.pad = pad; g->p.taps = op.k * op.k;
    g->p.cblocks = op.cout / 64;
    g->p.ntap_ch = op.cin;
    g->p.ntap = cls[q].n;
    for (int t = 0; t < cls[q].n; ++t) {
      g->p.tap_rs[t] = cls[q].rs[t];
      g->p.tap_dh[t] = cls[q].dh[t];
      g->p.tap_dw[t] = cls[q].dw[t];
    }
    if (st == 2) {
      g->p.ostride = 2; g->p.py = q / 2; g->p.px = q % 2;
      g->p.Hq = Ho; g->p.Wq = Wo; g->p.oH = a.H; g->p.oW = a.W;
    }
    const int M = o.N * Ho * Wo, KB = cls[q].n * g->p.cblocks;
    choose_tiles(c, g, M, op.cin, KB, op.cin);
    if (!map_window(&g->p.tmA, o.grad, o.N, Ho, Wo, o.C, Wo, rows, imgs) ||
        !map_2d(&g->p.tmB, w, op.cout, int64_t(g->p.taps) * op.cin, BK)) {
      delete g;
      for (TcGemm* x : *out) (void)x;
      out->clear();
      return false;
    }
    CUtensorMap cb;
    if (map_chunked(&cb, w, op.cout, int64_t(g->p.taps) * op.cin, BK, g->bn / 64)) { g->p.tmB = cb; g->p.chunk_b = 1; }
    if (!finish(c, g, M, op.cin, double(cls[q].n) * op.cout)) {
      out->clear();
      return false;
    }
    out->push_back(g);
  }
  return true;
}

TcGemm* tc_plan_wgrad(TcContext* c, fo_server* s, int i) {
  if (!c || !bf16_server(s) || getenv("FO_NO_TC")) return nullptr;
  const fo_op& op = s->ops[i];
  const Tensor& a = s->T[op.in0];
  const Tensor& o = s->T[i + 1];
  if (o.dt != kBF16) return nullptr;
  TcGemm* g = new TcGemm();
  g->p.out = s->grad + s->segs[s->op_segs[i][0]].off;
  g->p.out_f32 = 1;
  if (plain_gemm(op)) {
    if (!plain_gemm_ok(op)) { delete g; return nullptr; }
    g->kind = LIN_WGRAD;
    g->name = op.kind == FO_OP_LINEAR ? "tc_linear_wgrad" : "tc_conv1x1_wgrad";
    g->p.ldo = op.cin;
    int rows = int(a.rows()), KB = (rows + BK - 1) / BK;
    choose_tiles(c, g, op.cout, op.cin, KB, op.cin);
    g->input_B = s->T[op.in0].is_input();
    if (!map_2d(&g->p.tmA, o.grad, rows, op.cout, BK)) { delete g; return nullptr; }
    CUtensorMap ca;
    if (map_chunked(&ca, o.grad, rows, op.cout, BK, BM / 64)) { g->p.tmA = ca; g->p.chunk_a = 1; }
    const int nchunk = g->bn / 64;
    g->p.chunk_b = op.cin % 64 == 0 ? 1 : 0;
    auto map_b = [&](CUtensorMap* m, const void* base) {
      if (g->p.chunk_b && map_chunked(m, base, rows, op.cin, BK, nchunk)) return true;
      g->p.chunk_b = 0;
      return map_2d(m, base, rows, op.cin, BK);
    };
    if (g->input_B) {
      g->slot_maps.resize(s->cfg.omega);
      for (int pass = 0; pass < 2; ++pass) {   // a second pass if chunked maps fell back midway
        const int chunked = g->p.chunk_b;
        for (int sl = 0; sl < s->cfg.omega; ++sl)
          if (!map_b(&g->slot_maps[sl], s->slab + size_t(sl) * s->slot_stride)) { delete g; return nullptr; }
        if (chunked == g->p.chunk_b) break;
      }
    } else if (!map_b(&g->p.tmB, tensor_act(s, op.in0))) { delete g; return nullptr; }
    return finish(c, g, op.cout, op.cin, double(rows));
  }
  const int st = op.stride, Ho = o.H, Wo = o.W;
  if (op.cin % 64 || op.cout % 128 || (st == 2 && (a.H != 2 * Ho || a.W != 2 * Wo))) { delete g; return nullptr; }
  int rows, imgs;
  if (!window_ok(a.N, Ho, Wo, BK, &rows, &imgs) || (int64_t(a.N) * Ho * Wo) % BK) { delete g; return nullptr; }
  g->kind = CONV_WGRAD;
  g->name = "tc_conv_wgrad";
  g->p.ldo = op.k * op.k * op.cin;
  g->p.H = Ho; g->p.W = Wo; g->p.ksz = op.k; g->p.pad = op.k / 2; g->p.taps = op.k * op.k; g->p.stride = st;
  g->p.ntap_ch = op.cin;
  int P = a.N * Ho * Wo, KB = P / BK;
  int N = g->p.taps * op.cin;
  choose_tiles(c, g, op.cout, N, KB, op.cin);
  g->input_B = s->T[op.in0].is_input();
  if (!map_2d(&g->p.tmA, o.grad, P, op.cout, BK)) { delete g; return nullptr; }
  CUtensorMap ca;
  if (map_chunked(&ca, o.grad, P, op.cout, BK, BM / 64)) { g->p.tmA = ca; g->p.chunk_a = 1; }
  const int nchunk = std::min(g->bn, op.cin) / 64;   // channel chunks per box (one box per tap)
  g->p.chunk_b = 1;
  auto map_b = [&](CUtensorMap* m, const void* base) {
    if (g->p.chunk_b && map_window_chunked(m, base, a.N, a.H, a.W, a.C, Wo, rows, imgs, st, nchunk)) return true;
    g->p.chunk_b = 0;
    return map_window(m, base, a.N, a.H, a.W, a.C, Wo, rows, imgs, st);
  };
  if (g->input_B) {
    g->slot_maps.resize(s->cfg.omega);
    for (int pass = 0; pass < 2; ++pass) {   // a second pass if chunked maps fell back midway
      const int chunked = g->p.chunk_b;
      for (int sl = 0; sl < s->cfg.omega; ++sl)
        if (!map_b(&g->slot_maps[sl], s->slab + size_t(sl) * s->slot_stride)) { delete g; return nullptr; }
      if (chunked == g->p.chunk_b) break;
    }
  } else if (!map_b(&g->p.tmB, tensor_act(s, op.in0))) { delete g; return nullptr; }
  return finish(c, g, op.cout, N, double(P));
}

void tc_run(TcGemm* g, const void* input, cudaStream_t st) {
  (void)input;
  TcContext* c = g->ctx;
  if (g->input_A) g->p.tmA = g->slot_maps[c->slot];
  if (g->input_B) g->p.tmB = g->slot_maps[c->slot];
  if (g->input_acc) g->p.accsrc = static_cast<const bf16*>(c->s->cur_in);
  if (g->splits == 1) {
    launch_k(g->fn, g->grid, kPersistThreads, g->smem, st, g->p);
    return;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = g->grid;
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = g->smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = g->splits;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 2 : 1;
  cudaLaunchKernelEx(&cfg, g->fn, g->p);
}

int tc_splits(const TcGemm* g) { return g->splits; }
double tc_flops(const TcGemm* g) { return g->flops; }

const char* tc_name(const TcGemm* g) { return g->name; }

}  // namespace fo
