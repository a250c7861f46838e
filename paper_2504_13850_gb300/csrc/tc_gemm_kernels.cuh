// Tensor-core GEMM / implicit-GEMM convolution for sm_103a: tcgen05.mma
// (kind::f16, bf16 operands, fp32 accumulator in TMEM) fed by TMA tiles in
// 128-byte-swizzled shared memory, with a warp-specialised pipeline:
//   warp 0      TMA producer (one thread)
//   warp 1      TMEM allocator and MMA issuer (one thread)
//   epilogue    tcgen05.ld of the 128 x BN accumulator, then the bias /
//               ReLU / ReLU mask / residual add and the bf16 or fp32 store
//               (four warps in the split-K kernel, eight in the persistent one)
// Every mbarrier wait is bounded: on timeout the kernel records an error
// code in global memory and leaves instead of spinning forever.
//
// Problem kinds (D[M][N] = sum_k A[M][k] B[N][k]):
//   LIN_FWD    Y = X W^T          A = X  [rows][cin] K-major,  B = W [cout][cin] K-major
//   LIN_DGRAD  dX = dY W          A = dY [rows][cout] K-major, B = W (N = cin contiguous) MN-major
//   LIN_WGRAD  dW = dY^T X        A = dY (M = cout contiguous) MN-major, B = X MN-major
//   CONV_FPROP y = conv(x, W)     A = x window (per tap, 4-D TMA with zero fill) K-major,
//                                 B = W [Co][taps*Ci] K-major
//   CONV_DGRAD dx = conv^T(dy, W) A = dy window, taps shifted the other way,
//                                 B = W rows co, columns tap*Ci + ci: MN-major
//   CONV_WGRAD dW = sum_p dy (x) x-window: A = dy [P][Co] MN-major, B = x window MN-major
#pragma once
#include "fo_common.cuh"
#include "fo_ptx.cuh"

#include <cuda.h>
#include <cstdint>

namespace fo {
namespace tcg {

enum Kind { LIN_FWD = 0, LIN_DGRAD = 1, LIN_WGRAD = 2, CONV_FPROP = 3, CONV_DGRAD = 4, CONV_WGRAD = 5 };

// Epilogue variants, fixed at compile time so that each kernel carries only
// the code of its own epilogue (the epilogue runs once per tile from a cold
// instruction cache, so unused branches cost time even when not taken).
// The bias is applied when present (zeros otherwise).
enum Epi : int {
  E_RELU = 1,   // y = max(y, 0)
  E_MASK = 2,   // ReLU mask of the input-gradient: y = 0 where mask <= 0
  E_ACC = 4,    // y += accsrc (accumulate, or a residual add into a new buffer)
  E_F32 = 8,    // fp32 output, nothing else (the weight gradients)
  E_POOL = 16,  // with E_RELU: a 2x2 max-pool of the conv output (pool_w <= 16
                // columns per image row, so a warp's 32 rows hold whole
                // windows); writes the pooled values and the window codes
                // instead of the full-resolution output
  E_GELU = 64,  // with E_TMA: out = the bias-added result (bf16), and
                // gelu_out = GELU of that stored value (the FFN's activation)
  E_TMA = 32,   // persistent kernel, bf16 row-major output: the accumulator
                // starts from the bias (and, for E_ACC without E_MASK, the
                // accumulate operand), written into tensor memory before the
                // tile's MMAs, and each 32 x 32 chunk leaves through shared
                // memory by a TMA tensor store (tmO)
};

constexpr int BM = 128;      // UMMA M (cta_group::1)
constexpr int BK = 64;       // k-block: one 128-byte swizzle row of bf16
constexpr int UK = 16;       // UMMA K for kind::f16
constexpr int kThreads = 192;
constexpr int kSmemBudget = 200 * 1024;

struct TcParams;
typedef void (*KernelFn)(const TcParams);

struct TcParams {
  CUtensorMap tmA;
  CUtensorMap tmB;
  CUtensorMap tmO;      // E_TMA: the output, bf16 [M][ldo], box 32 x 32, 64-byte swizzle
  CUtensorMap tmG;      // E_GELU: gelu_out, the same layout
  int M, N, KB, kper;
  // window geometry (spatial size of the windowed tensor and its taps)
  int H, W, ksz, pad, taps;
  int stride;           // CONV_FPROP / CONV_WGRAD: stride of the windowed input
  int cblocks;          // 64-channel blocks per tap (contraction channels)
  int ntap_ch;          // CONV_WGRAD / CONV_DGRAD: channels per tap in the N index (Ci)
  int win_rows, win_imgs;  // rows/images covered by one window box
  // CONV_DGRAD: the taps of this output-parity class, as (tap index r*k+s,
  // row shift, column shift) of the gradient window
  int ntap;
  int tap_rs[9], tap_dh[9], tap_dw[9];
  // output rows: GEMM row m = (n, i, j) over an Hq x Wq grid is written to
  // row (n*oH + ostride*i + py)*oW + ostride*j + px of `out` (identity when
  // ostride == 0)
  int ostride, py, px, Hq, Wq, oH, oW;
  // MN-major operands whose 64-wide chunks one TMA box brings in at once
  // (a chunk dimension of stride 128 bytes as the box's outermost dimension)
  int chunk_a, chunk_b;
  // epilogue
  void* out;
  int ldo;
  const float* bias;
  const bf16* mask;     // ReLU mask (same layout as out): keep where mask > 0
  int relu, acc, out_f32;
  int tma_out;          // E_TMA (tmO is valid)
  bf16* gelu_out;       // E_GELU
  // bf16 outputs only: the accumulate operand (acc) is read from accsrc, which
  // is `out` itself unless the sum goes to a new buffer (a residual add:
  // out = result + accsrc).
  const bf16* accsrc;
  // E_POOL: pooled output [N][H/2][W/2][ldo] and the position of each
  // window's first maximum (0..3, row-major) per pooled element; pool_w is the
  // output image width W (GEMM rows are (n, h, w) with h, w the image row and
  // column)
  bf16* pool_out;
  uint8_t* pool_code;
  int pool_w;
  int* err;
  // split-K: fp32 partial tiles, [tile][rank][BN/32][8][BM] float4 (tile =
  // blockIdx.y * gridDim.x + blockIdx.x); only rows a rank does not own are written
  float* ws;
};

__device__ __forceinline__ size_t out_row(const TcParams& p, int m) {
  if (!p.ostride) return size_t(m);
  const int hw = p.Hq * p.Wq;
  const int n = m / hw, rem = m % hw, i = rem / p.Wq, j = rem % p.Wq;
  return (size_t(n) * p.oH + p.ostride * i + p.py) * p.oW + p.ostride * j + p.px;
}

// Pooled row of window `win` (0..7) of the 32 GEMM rows from m_base (m_base a
// multiple of 2 W, so the rows are whole image rows starting at an even one),
// and the GEMM row (offset from m_base) of the window's top-left position.
__device__ __forceinline__ void pool_window(const TcParams& p, int m_base, int win, size_t* prow, int* r0) {
  const int W = p.pool_w, wp = W / 2;
  const int hp = win / wp, wq = win % wp;
  *r0 = 2 * hp * W + 2 * wq;
  *prow = (size_t(m_base / W) / 2 + hp) * wp + wq;
}

// Epilogue of 32 consecutive outputs (m, n..n+31) held by one thread: bias,
// ReLU, ReLU mask, accumulate, store as fp32 or bf16 (16-byte accesses).
// `sbias`: shared-memory address of the bias values for columns n..n+31.
// Columns >= N (the ragged last tile; N is a multiple of 8) are not touched.
// bf16 outputs take their ReLU-mask and accumulate operands preloaded by
// load_row32 (so that a caller can fetch them ahead of time).
template <int EPI>
__device__ __forceinline__ void load_row32(const TcParams& p, int m_gemm, int n, uint4 (&mk)[4], uint4 (&ac)[4]) {
  if constexpr ((EPI & E_F32) || !(EPI & (E_MASK | E_ACC))) return;
  const int nv = p.N - n;
  if (nv <= 0 || m_gemm >= p.M) return;
  const size_t m = out_row(p, m_gemm);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (8 * j >= nv) break;
    if constexpr (EPI & E_MASK) mk[j] = *reinterpret_cast<const uint4*>(p.mask + m * p.ldo + n + 8 * j);
    if constexpr (EPI & E_ACC) ac[j] = *reinterpret_cast<const uint4*>(p.accsrc + m * p.ldo + n + 8 * j);
  }
}
template <int EPI>
__device__ __forceinline__ void store_row32(const TcParams& p, int m_gemm, int n, float (&v)[32], uint32_t sbias,
                                            const uint4 (&mk)[4], const uint4 (&ac)[4]) {
  const size_t m = out_row(p, m_gemm);
  const int nv = p.N - n;   // valid columns from n
  if (nv <= 0) return;
  if constexpr (EPI & E_F32) {   // a weight gradient: plain fp32 store
    float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(p.out) + m * p.ldo + n);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (4 * j >= nv) break;
      dst[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) {   // zeros without a bias
      const float4 b = ld_shared4(sbias + 16u * j);
      v[4 * j] += b.x; v[4 * j + 1] += b.y; v[4 * j + 2] += b.z; v[4 * j + 3] += b.w;
    }
    if constexpr (EPI & E_RELU)
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = fmaxf(v[j], 0.f);
    uint4* dst = reinterpret_cast<uint4*>(reinterpret_cast<bf16*>(p.out) + m * p.ldo + n);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (8 * j >= nv) break;
      if constexpr (EPI & E_MASK) {
        const bf16* e = reinterpret_cast<const bf16*>(&mk[j]);
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (!(__bfloat162float(e[q]) > 0.f)) v[8 * j + q] = 0.f;
      }
      if constexpr (EPI & E_ACC) {
        const bf16* ob = reinterpret_cast<const bf16*>(&ac[j]);
#pragma unroll
        for (int e = 0; e < 8; ++e) v[8 * j + e] += __bfloat162float(ob[e]);
      }
      uint4 pk;
      uint32_t* pw = reinterpret_cast<uint32_t*>(&pk);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        __nv_bfloat162 h2 = __floats2bfloat162_rn(v[8 * j + 2 * e], v[8 * j + 2 * e + 1]);
        pw[e] = *reinterpret_cast<uint32_t*>(&h2);
      }
      dst[j] = pk;
    }
  }
}

// E_POOL in the split-K owner: lane = GEMM row m_base + lane with its 32
// columns v (bias and ReLU applied); the 2 x 2 windows are lanes {l, l ^ 1,
// l ^ W, l ^ W ^ 1}, reduced with shuffles (first maximum in row-major
// window order), and the window's top-left lane stores the pooled values and
// codes.  Every lane of the warp must call it.
template <int EPI>
__device__ __forceinline__ void pool_row32(const TcParams& p, int m_base, int lane, int n, const float (&v)[32]) {
  const int W = p.pool_w;
  const int pos = ((lane / W) & 1) * 2 + (lane & 1);   // this lane's place in its window
  float mx[32];
  uint32_t cd[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    float m = fmaxf(v[j], __shfl_xor_sync(0xffffffffu, v[j], 1));
    m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, W));
    int c = v[j] == m ? pos : 4;
    c = min(c, __shfl_xor_sync(0xffffffffu, c, 1));
    c = min(c, __shfl_xor_sync(0xffffffffu, c, W));
    mx[j] = m;
    cd[j / 4] |= uint32_t(c) << (8 * (j % 4));
  }
  if (pos != 0) return;   // the window's top-left lane stores
  const int hp = (lane / W) / 2, wq = (lane % W) / 2;
  const size_t prow = (size_t(m_base / W) / 2 + hp) * (W / 2) + wq;
  const int nv = p.N - n;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (8 * j >= nv) break;
    uint4 pk;
    uint32_t* pw = reinterpret_cast<uint32_t*>(&pk);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      __nv_bfloat162 h2 = __floats2bfloat162_rn(mx[8 * j + 2 * q], mx[8 * j + 2 * q + 1]);
      pw[q] = *reinterpret_cast<uint32_t*>(&h2);
    }
    *reinterpret_cast<uint4*>(p.pool_out + prow * p.ldo + n + 8 * j) = pk;
    *reinterpret_cast<uint2*>(p.pool_code + prow * p.ldo + n + 8 * j) = make_uint2(cd[2 * j], cd[2 * j + 1]);
  }
}

// Coalesced epilogue of a 32-row x 32-column accumulator chunk held one row
// per lane (lane = row, r[j] = column j).  The warp stages the chunk in its
// 4 KB shared-memory buffer (16-byte units XOR-swizzled by row, so both the
// row-wise writes and the column-wise reads are free of bank conflicts), then
// reads it back so that consecutive lanes own consecutive columns of a row:
// bias, ReLU, ReLU mask, accumulate and the stores then touch whole 32-byte
// sectors (bf16: 8 rows x 64 B per instruction; fp32: 4 rows x 128 B).
// The bias values lane `lane` applies in epilogue_chunk32 for the chunk at
// column n: 8 columns from 8 * (lane % 4) (bf16 outputs; zeros without a
// bias, and for the fp32 weight gradients, which have none).
template <int EPI>
__device__ __forceinline__ void load_bias8(const TcParams& p, int lane, int n, float (&b)[8]) {
  float4 b0 = make_float4(0.f, 0.f, 0.f, 0.f), b1 = b0;
  if constexpr (!(EPI & E_F32)) {
    if (p.bias && n + 8 * (lane & 3) < p.N) {
      const float4* src = reinterpret_cast<const float4*>(p.bias + n);
      b0 = __ldg(src + 2 * (lane & 3));
      b1 = __ldg(src + 2 * (lane & 3) + 1);
    }
  }
  b[0] = b0.x; b[1] = b0.y; b[2] = b0.z; b[3] = b0.w; b[4] = b1.x; b[5] = b1.y; b[6] = b1.z; b[7] = b1.w;
}

template <int EPI>
__device__ __forceinline__ void epilogue_chunk32(const TcParams& p, uint32_t stage, int lane, int m_base, int n,
                                                 const uint32_t (&r)[32], const float (&b)[8]) {
  // bf16 outputs: the chunk's ReLU-mask and accumulate operands (four rows
  // per lane) are loaded before the staging, all at once, so that their
  // latency overlaps the staging and each other instead of adding up row by
  // row (the dominant cost of an input-gradient epilogue otherwise).
  const int co = lane & 3;                   // bf16: columns 8co .. 8co+7
  uint4 mk[4] = {}, ac[4] = {};
  size_t off[4];
  bool ok[4];
  if constexpr (!(EPI & E_F32)) {
#pragma unroll
    for (int it = 0; it < 4; ++it) {
      const int mg = m_base + it * 8 + (lane >> 2);
      ok[it] = mg < p.M && n + 8 * co < p.N;
      off[it] = ok[it] ? out_row(p, mg) * p.ldo + n + 8 * co : 0;
      if constexpr (EPI & E_MASK)
        if (ok[it]) mk[it] = *reinterpret_cast<const uint4*>(p.mask + off[it]);
      if constexpr (EPI & E_ACC)
        if (ok[it]) ac[it] = *reinterpret_cast<const uint4*>(p.accsrc + off[it]);
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j)
    st_shared4(stage + 16u * (lane * 8 + (j ^ (lane & 7))), r[4 * j], r[4 * j + 1], r[4 * j + 2], r[4 * j + 3]);
  __syncwarp();
  if constexpr (EPI & E_POOL) {   // 2 x 2 max-pool of the chunk's 32 rows: lane = (window, 8 channels)
    const int win = lane >> 2;
    size_t prow;
    int r0;
    pool_window(p, m_base, win, &prow, &r0);
    if (n + 8 * co < p.N) {
      float best[8];
      int arg[8];
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int rr = r0 + (t >> 1) * p.pool_w + (t & 1);
        const float4 v0 = ld_shared4(stage + 16u * (rr * 8 + ((2 * co) ^ (rr & 7))));
        const float4 v1 = ld_shared4(stage + 16u * (rr * 8 + ((2 * co + 1) ^ (rr & 7))));
        const float e[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const float x = fmaxf(e[q] + b[q], 0.f);   // bias and ReLU, then the window maximum
          if (t == 0 || x > best[q]) {
            best[q] = x;
            arg[q] = t;
          }
        }
      }
      uint4 pk;
      uint32_t* pw = reinterpret_cast<uint32_t*>(&pk);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        __nv_bfloat162 h2 = __floats2bfloat162_rn(best[2 * q], best[2 * q + 1]);
        pw[q] = *reinterpret_cast<uint32_t*>(&h2);
      }
      const size_t off = prow * p.ldo + n + 8 * co;
      *reinterpret_cast<uint4*>(p.pool_out + off) = pk;
      *reinterpret_cast<uint2*>(p.pool_code + off) =
          make_uint2(uint32_t(arg[0]) | uint32_t(arg[1]) << 8 | uint32_t(arg[2]) << 16 | uint32_t(arg[3]) << 24,
                     uint32_t(arg[4]) | uint32_t(arg[5]) << 8 | uint32_t(arg[6]) << 16 | uint32_t(arg[7]) << 24);
    }
  } else if constexpr (EPI & E_F32) {   // a weight gradient: plain fp32 store, 4 rows x 128 B per instruction
    const int cq = lane & 7;     // 16-byte unit: columns 4cq .. 4cq+3
#pragma unroll 1
    for (int it = 0; it < 8; ++it) {
      const int rr = it * 4 + (lane >> 3);
      const int mg = m_base + rr;
      const float4 v = ld_shared4(stage + 16u * (rr * 8 + (cq ^ (rr & 7))));
      if (mg < p.M && n + 4 * cq < p.N)
        reinterpret_cast<float4*>(reinterpret_cast<float*>(p.out) + out_row(p, mg) * p.ldo + n)[cq] = v;
    }
  } else {
#pragma unroll
    for (int it = 0; it < 4; ++it) {
      const int rr = it * 8 + (lane >> 2);
      const float4 v0 = ld_shared4(stage + 16u * (rr * 8 + ((2 * co) ^ (rr & 7))));
      const float4 v1 = ld_shared4(stage + 16u * (rr * 8 + ((2 * co + 1) ^ (rr & 7))));
      if (ok[it]) {
        float e[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
        for (int q = 0; q < 8; ++q) e[q] += b[q];
        if constexpr (EPI & E_RELU)
#pragma unroll
          for (int q = 0; q < 8; ++q) e[q] = fmaxf(e[q], 0.f);
        if constexpr (EPI & E_MASK) {
          const bf16* mkp = reinterpret_cast<const bf16*>(&mk[it]);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (!(__bfloat162float(mkp[q]) > 0.f)) e[q] = 0.f;
        }
        if constexpr (EPI & E_ACC) {
          const bf16* eo = reinterpret_cast<const bf16*>(&ac[it]);
#pragma unroll
          for (int q = 0; q < 8; ++q) e[q] += __bfloat162float(eo[q]);
        }
        uint4 pk;
        uint32_t* pw = reinterpret_cast<uint32_t*>(&pk);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          __nv_bfloat162 h2 = __floats2bfloat162_rn(e[2 * q], e[2 * q + 1]);
          pw[q] = *reinterpret_cast<uint32_t*>(&h2);
        }
        *reinterpret_cast<uint4*>(reinterpret_cast<bf16*>(p.out) + off[it]) = pk;
      }
    }
  }
  __syncwarp();
}

template <int KIND>
struct KindTraits {
  static constexpr bool a_mn = (KIND == LIN_WGRAD || KIND == CONV_WGRAD);
  static constexpr bool b_mn = (KIND == LIN_DGRAD || KIND == LIN_WGRAD || KIND == CONV_DGRAD || KIND == CONV_WGRAD);
};

// Issue the TMA loads of k-block `kb` for output tile (m0, n0).
template <int KIND, int BN>
__device__ __forceinline__ void load_kblock(const TcParams& p, int kb, int m0, int n0, char* sa, char* sb,
                                            uint64_t* bar) {
  const int HW = p.H * p.W;
  if (KIND == LIN_FWD || KIND == LIN_DGRAD) {
    tma_2d(sa, &p.tmA, bar, kb * BK, m0);
  } else if (KIND == LIN_WGRAD || KIND == CONV_WGRAD) {
    if (p.chunk_a)
      tma_3d(sa, &p.tmA, bar, 0, kb * BK, m0 / 64);
    else
#pragma unroll
      for (int j = 0; j < BM / 64; ++j) tma_2d(sa + j * BK * 128, &p.tmA, bar, m0 + j * 64, kb * BK);
  } else if (KIND == CONV_FPROP) {  // windowed A over the (strided) input
    const int tap = kb / p.cblocks, c0 = (kb % p.cblocks) * 64;
    const int r = tap / p.ksz, s = tap % p.ksz;
    const int n_img = m0 / HW, h0 = (m0 % HW) / p.W;   // H, W: output grid
    tma_4d(sa, &p.tmA, bar, c0, s - p.pad, h0 * p.stride + r - p.pad, n_img);
  } else {  // CONV_DGRAD: window over the output gradient, shifted per tap
    const int t = kb / p.cblocks, c0 = (kb % p.cblocks) * 64;
    const int n_img = m0 / HW, h0 = (m0 % HW) / p.W;   // H, W: the class grid (= gradient grid)
    tma_4d(sa, &p.tmA, bar, c0, p.tap_dw[t], h0 + p.tap_dh[t], n_img);
  }
  if (KIND == LIN_FWD) {
    tma_2d(sb, &p.tmB, bar, kb * BK, n0);
  } else if (KIND == CONV_FPROP) {
    const int tap = kb / p.cblocks, c0 = (kb % p.cblocks) * 64;
    tma_2d(sb, &p.tmB, bar, tap * p.ntap_ch + c0, n0);
  } else if (KIND == LIN_DGRAD || KIND == LIN_WGRAD) {
    if (p.chunk_b)
      tma_3d(sb, &p.tmB, bar, 0, kb * BK, n0 / 64);
    else
#pragma unroll
      for (int j = 0; j < BN / 64; ++j) tma_2d(sb + j * BK * 128, &p.tmB, bar, n0 + j * 64, kb * BK);
  } else if (KIND == CONV_DGRAD) {
    const int t = kb / p.cblocks, co0 = (kb % p.cblocks) * 64;
    const int tap = p.tap_rs[t];
    if (p.chunk_b)
      tma_3d(sb, &p.tmB, bar, 0, co0, (tap * p.ntap_ch + n0) / 64);
    else
#pragma unroll
      for (int j = 0; j < BN / 64; ++j) tma_2d(sb + j * BK * 128, &p.tmB, bar, tap * p.ntap_ch + n0 + j * 64, co0);
  } else if (p.chunk_b) {  // CONV_WGRAD: the tile's channel chunks in one box per tap
    // (a tile wider than Ci spans BN / Ci taps; a ragged last tile's tap past
    // the last one loads a shifted window whose columns the epilogue drops)
    const int cw = BN < p.ntap_ch ? BN : p.ntap_ch;
    const int pix0 = kb * BK;
    const int n_img = pix0 / HW, h0 = (pix0 % HW) / p.W;
    for (int t = 0; t * cw < BN; ++t) {
      const int nn = n0 + t * cw;
      const int tap = nn / p.ntap_ch, ci0 = nn % p.ntap_ch;
      const int r = tap / p.ksz, s = tap % p.ksz;
      tma_5d(sb + t * (cw / 64) * BK * 128, &p.tmB, bar, 0, s - p.pad, h0 * p.stride + r - p.pad, n_img, ci0 / 64);
    }
  } else {  // CONV_WGRAD: N index = tap * Ci + ci; K = output pixel
    const int pix0 = kb * BK;
    const int n_img = pix0 / HW, h0 = (pix0 % HW) / p.W;   // H, W: output grid
#pragma unroll
    for (int j = 0; j < BN / 64; ++j) {
      const int nn = n0 + j * 64;
      const int tap = nn / p.ntap_ch, ci = nn % p.ntap_ch;
      const int r = tap / p.ksz, s = tap % p.ksz;
      tma_4d(sb + j * BK * 128, &p.tmB, bar, ci, s - p.pad, h0 * p.stride + r - p.pad, n_img);
    }
  }
}

// Split-K: the gridDim.z CTAs of a (1, 1, S) cluster each run k-blocks
// [kb0, kb0 + kper) of the same output tile.  Rank z owns the 32-column
// chunks [z*NC/S, (z+1)*NC/S) of the tile (NC = BN/32), all 128 rows, so all
// four epilogue warps of every CTA take part.  After the MMAs every CTA
// writes the chunks it does not own from TMEM to its slice of a global fp32
// workspace (L2-resident; each warp store covers 512 contiguous bytes); the
// cluster barrier (release / acquire) orders those writes before the owners'
// reads; each owner pulls the other ranks' slices of its chunks into its idle
// pipeline buffers with bulk copies, adds the S partials in rank order
// (deterministic) and runs the epilogue, with the ReLU-mask / accumulate
// operands of the next chunk loaded while the current one is stored.
// (Distributed-shared-memory stores moved these partials at only ~20 GB/s
// per SM pair, and an owner that read them chunk by chunk from L2 waited a
// full round trip per chunk.)
template <int KIND, int BN, int STAGES, int EPI>
__global__ void __launch_bounds__(kThreads, 1) tc_gemm_kernel(const __grid_constant__ TcParams p) {
  extern __shared__ __align__(1024) char smem_raw[];
  char* smem = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  constexpr int A_BYTES = BM * BK * 2;
  constexpr int B_BYTES = BN * BK * 2;
  constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* accum = empty + STAGES;
  uint64_t* rbar = accum + 1;   // the owner's bulk copies of the other ranks' partials
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(rbar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* sbias = reinterpret_cast<float*>(smem + STAGES * STAGE_BYTES + 256);   // bias[n0 .. n0 + BN)
  static_assert(STAGES * STAGE_BYTES + 1024 + 256 + 4 * BN <= 232448, "shared memory per CTA");
  static_assert(2 * STAGES * 8 + 8 + 8 + 4 + 4 <= 256, "barrier area");

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM;
  const int S = gridDim.z, me = blockIdx.z;
  const int kb0 = me * p.kper;
  const int kb1 = min(p.KB, kb0 + p.kper);
  const int nk = kb1 - kb0;
  constexpr int NC = BN / 32;
  const int c0 = me * NC / S, c1 = (me + 1) * NC / S;   // owned 32-column chunks
  constexpr uint32_t kCols = BN < 32 ? 32 : BN;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accum, 1);
    mbar_init(rbar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmB)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();   // every block of this kernel is resident and holds its tensor memory
  pdl_wait();      // the previous kernel's writes are visible from here on

  if (warp == 0) {
    if (lane == 0) {
      for (int it = 0; it < nk; ++it) {
        const int s = it % STAGES;
        if (!mbar_wait(&empty[s], ((it / STAGES) & 1) ^ 1)) {
          atomicExch(p.err, 1);
          *abort_flag = 1;
          break;
        }
        if (*abort_flag) break;
        char* sa = smem + s * STAGE_BYTES;
        mbar_expect_tx(&full[s], STAGE_BYTES);
        load_kblock<KIND, BN>(p, kb0 + it, m0, n0, sa, sa + A_BYTES, &full[s]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = instr_desc(BN, KindTraits<KIND>::a_mn, KindTraits<KIND>::b_mn);
      bool ok = true;
      for (int it = 0; it < nk; ++it) {
        const int s = it % STAGES;
        if (!mbar_wait(&full[s], (it / STAGES) & 1)) {
          atomicExch(p.err, 2);
          *abort_flag = 1;
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = smem_u32(smem + s * STAGE_BYTES);
        const uint32_t b0 = a0 + A_BYTES;
#pragma unroll
        for (int k = 0; k < BK / UK; ++k) {
          uint64_t ad, bd;
          if (KindTraits<KIND>::a_mn) ad = smem_desc(a0 + k * UK * 128, BK * 128, 1024);
          else ad = smem_desc(a0 + k * UK * 2, 16, 1024);
          if (KindTraits<KIND>::b_mn) bd = smem_desc(b0 + k * UK * 128, BK * 128, 1024);
          else bd = smem_desc(b0 + k * UK * 2, 16, 1024);
          mma_f16(tmem, ad, bd, idesc, (it > 0 || k > 0) ? 1u : 0u);
        }
        mma_commit(&empty[s]);
      }
      if (ok) mma_commit(accum);
      else mbar_expect_tx(accum, 0);  // release the epilogue without data
    }
  } else {
    // the tile's bias into shared memory while the MMAs run
    for (int j = threadIdx.x - 64; j < BN; j += 128) sbias[j] = p.bias && n0 + j < p.N ? p.bias[n0 + j] : 0.f;
    if (!mbar_wait(accum, 0)) atomicExch(p.err, 3);
    tc_fence_after();
  }
  // Chunks this CTA does not own go to its slice of the workspace:
  // ws_tile[rank][chunk][j][row] (float4), one 16 KB slice per (rank, chunk).
  constexpr int SLICE = 8 * BM;   // float4 per slice
  const size_t tile = size_t(blockIdx.y) * gridDim.x + blockIdx.x;
  float4* ws_tile = reinterpret_cast<float4*>(p.ws) + tile * size_t(S) * NC * SLICE;
  const int q = warp % 4, row = q * 32 + lane;
  const uint32_t trow = tmem + (uint32_t(q * 32) << 16);
  if (warp >= 2) {
    float4* dst = ws_tile + size_t(me) * NC * SLICE + row;
#pragma unroll 1
    for (int c = 0; c < NC; ++c) {
      if (c >= c0 && c < c1) continue;
      uint32_t r[32];
      tmem_ld32(trow + uint32_t(32 * c), r);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        __stcg(dst + (c * 8 + j) * BM,
               make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]), __uint_as_float(r[4 * j + 2]),
                           __uint_as_float(r[4 * j + 3])));
    }
  }
  // Every CTA's partials are written (release) and visible (acquire).
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const int nown = c1 - c0;
  float4* recv = reinterpret_cast<float4*>(smem);   // [(rank, chunk)][j][row]: the idle pipeline buffers
  auto recv_slot = [&](int z, int c) { return (z < me ? z : z - 1) * nown + (c - c0); };
  if (threadIdx.x == 64 && nown > 0) {
    asm volatile("fence.proxy.async;" ::: "memory");   // peers' generic writes before these async-proxy reads
    mbar_expect_tx(rbar, uint32_t((S - 1) * nown * SLICE * 16));
    for (int z = 0; z < S; ++z) {
      if (z == me) continue;
      for (int c = c0; c < c1; ++c)
        bulk_g2s(recv + size_t(recv_slot(z, c)) * SLICE, ws_tile + (size_t(z) * NC + c) * SLICE, SLICE * 16, rbar);
    }
  }
  if (warp >= 2 && nown > 0) {
    const int mg = m0 + row;
    uint4 mk[4] = {}, ac[4] = {}, mk2[4] = {}, ac2[4] = {};
    load_row32<EPI>(p, mg, n0 + 32 * c0, mk, ac);
    if (!mbar_wait(rbar, 0)) atomicExch(p.err, 9);
#pragma unroll 1
    for (int c = c0; c < c1; ++c) {
      if (c + 1 < c1) load_row32<EPI>(p, mg, n0 + 32 * (c + 1), mk2, ac2);
      uint32_t r[32];
      tmem_ld32(trow + uint32_t(32 * c), r);
      if (mg < p.M || (EPI & E_POOL)) {   // a pooled conv has M % 128 == 0: every lane takes part
        float v[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = 0.f;
#pragma unroll 1
        for (int z = 0; z < S; ++z) {
          if (z == me) {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] += __uint_as_float(r[j]);
          } else {
            const uint32_t src = smem_u32(recv + size_t(recv_slot(z, c)) * SLICE + row);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float4 w = ld_shared4(src + uint32_t(j * BM * 16));
              v[4 * j] += w.x; v[4 * j + 1] += w.y; v[4 * j + 2] += w.z; v[4 * j + 3] += w.w;
            }
          }
        }
        if constexpr (EPI & E_POOL) {
          const uint32_t sb = smem_u32(sbias) + uint32_t(32 * c) * 4u;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 bb = ld_shared4(sb + 16u * j);
            v[4 * j] = fmaxf(v[4 * j] + bb.x, 0.f);
            v[4 * j + 1] = fmaxf(v[4 * j + 1] + bb.y, 0.f);
            v[4 * j + 2] = fmaxf(v[4 * j + 2] + bb.z, 0.f);
            v[4 * j + 3] = fmaxf(v[4 * j + 3] + bb.w, 0.f);
          }
          pool_row32<EPI>(p, m0 + q * 32, lane, n0 + 32 * c, v);
        } else {
          store_row32<EPI>(p, mg, n0 + 32 * c, v, smem_u32(sbias) + uint32_t(32 * c) * 4u, mk, ac);
        }
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        mk[j] = mk2[j];
        ac[j] = ac2[j];
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kCols) : "memory");
  }
}


// Persistent variant (no K split): gridDim.x CTAs loop over the output tiles
// (n fastest).  The TMA producer runs ahead across tile boundaries and the
// accumulator is double-buffered in TMEM, so the epilogue of one tile
// overlaps the MMAs of the next.  Barriers: full/empty per stage (TMA <->
// MMA), acc_full/acc_empty per accumulator (MMA <-> epilogue).
constexpr int kPersistThreads = 320;  // TMA warp, MMA warp, 8 epilogue warps
constexpr int kEpiStageBytes = 8 * 4096;  // one 32 x 32 fp32 staging buffer per epilogue warp
// E_TMA: the starting value of this thread's accumulator row m (TMEM lane
// address tbase), columns n_base .. n_base + CW - 1: the bias of each column,
// plus the accumulate operand unless a ReLU mask comes first (E_MASK | E_ACC
// adds it after the mask, in the epilogue); zeros outside the output.
template <int EPI, int CW>
__device__ __forceinline__ void tma_preload(const TcParams& p, uint32_t tbase, int m, int n_base) {
  const bool row_ok = m < p.M;
#pragma unroll 1
  for (int c = 0; c < CW; c += 32) {
    const int n = n_base + c;
    uint32_t v[32];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const bool col_ok = n + 8 * u < p.N;
      float4 b0 = make_float4(0.f, 0.f, 0.f, 0.f), b1 = b0;
      if (p.bias && col_ok) {
        b0 = __ldg(reinterpret_cast<const float4*>(p.bias + n + 8 * u));
        b1 = __ldg(reinterpret_cast<const float4*>(p.bias + n + 8 * u) + 1);
      }
      float e[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
      if constexpr ((EPI & E_ACC) && !(EPI & E_MASK)) {
        if (row_ok && col_ok) {
          const uint4 a = *reinterpret_cast<const uint4*>(p.accsrc + size_t(m) * p.ldo + n + 8 * u);
          const bf16* ab = reinterpret_cast<const bf16*>(&a);
#pragma unroll
          for (int j = 0; j < 8; ++j) e[j] += __bfloat162float(ab[j]);
        }
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) v[8 * u + j] = __float_as_uint(e[j]);
    }
    tmem_st32(tbase + uint32_t(c), v);
  }
}

// This thread's row (32 bf16, 16 packed words) into the 2 KB staging buffer
// `buf` in the layout of a 32 x 32 box of a 64-byte-swizzled map (row i at
// 64 i, its 16-byte unit u at u ^ ((i >> 1) & 3)).
__device__ __forceinline__ void stage_row64(uint32_t buf, int lane, const uint32_t (&pk)[16]) {
  const int f = (lane >> 1) & 3;
#pragma unroll
  for (int u = 0; u < 4; ++u)
    st_shared4(buf + 16u * uint32_t(lane * 4 + (u ^ f)), pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
}

// E_GELU: this thread's 32 accumulator values (bias included) as bf16 (the
// pre-activation, kept for the backward pass) and the GELU of each stored
// bf16 value, as the separate GELU kernel computes it.
__device__ __forceinline__ void gelu_pack32(const uint32_t (&r)[32], uint32_t (&hk)[16], uint32_t (&gk)[16]) {
#pragma unroll
  for (int q = 0; q < 16; ++q) {
    __nv_bfloat162 h2 = __floats2bfloat162_rn(__uint_as_float(r[2 * q]), __uint_as_float(r[2 * q + 1]));
    hk[q] = *reinterpret_cast<uint32_t*>(&h2);
    const float x0 = __low2float(h2), x1 = __high2float(h2);
    float c0, d0, c1, d1;
    normal_cdf_pdf(x0, c0, d0);
    normal_cdf_pdf(x1, c1, d1);
    __nv_bfloat162 g2 = __floats2bfloat162_rn(x0 * c0, x1 * c1);
    gk[q] = *reinterpret_cast<uint32_t*>(&g2);
  }
}

// E_TMA: one 32 x 32 chunk, this thread's row m and columns n .. n + 31 in
// r: ReLU / ReLU mask / accumulate after the mask, bf16, into the 2 KB
// staging buffer `buf` (512-byte aligned) in the layout of a 32 x 32 box of
// the 64-byte-swizzled output map (row i at 64 i, its 16-byte unit u at
// u ^ ((i >> 1) & 3)), made visible to the TMA store that follows.
template <int EPI>
__device__ __forceinline__ void tma_chunk32(const TcParams& p, uint32_t buf, int lane, int m, int n,
                                            const uint32_t (&r)[32]) {
  const bool row_ok = m < p.M;
  uint4 mk[4] = {}, ac[4] = {};
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const bool ok = row_ok && n + 8 * u < p.N;
    if constexpr (EPI & E_MASK)
      if (ok) mk[u] = *reinterpret_cast<const uint4*>(p.mask + size_t(m) * p.ldo + n + 8 * u);
    if constexpr ((EPI & E_ACC) && (EPI & E_MASK))
      if (ok) ac[u] = *reinterpret_cast<const uint4*>(p.accsrc + size_t(m) * p.ldo + n + 8 * u);
  }
  const int f = (lane >> 1) & 3;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    float e[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) e[j] = __uint_as_float(r[8 * u + j]);
    if constexpr (EPI & E_RELU)
#pragma unroll
      for (int j = 0; j < 8; ++j) e[j] = fmaxf(e[j], 0.f);
    if constexpr (EPI & E_MASK) {
      const bf16* mkp = reinterpret_cast<const bf16*>(&mk[u]);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (!(__bfloat162float(mkp[j]) > 0.f)) e[j] = 0.f;
      if constexpr (EPI & E_ACC) {
        const bf16* ap = reinterpret_cast<const bf16*>(&ac[u]);
#pragma unroll
        for (int j = 0; j < 8; ++j) e[j] += __bfloat162float(ap[j]);
      }
    }
    uint32_t pk[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      __nv_bfloat162 h2 = __floats2bfloat162_rn(e[2 * q], e[2 * q + 1]);
      pk[q] = *reinterpret_cast<uint32_t*>(&h2);
    }
    st_shared4(buf + 16u * uint32_t(lane * 4 + (u ^ f)), pk[0], pk[1], pk[2], pk[3]);
  }
  fence_proxy_async_smem();
}

template <int KIND, int BN, int STAGES, int EPI>
__global__ void __launch_bounds__(kPersistThreads, 1) tc_gemm_persistent(const __grid_constant__ TcParams p) {
  extern __shared__ __align__(1024) char smem_raw[];
  char* smem = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  constexpr int A_BYTES = BM * BK * 2;
  constexpr int B_BYTES = BN * BK * 2;
  constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static_assert(STAGES * STAGE_BYTES + kEpiStageBytes + 1024 + 256 <= 232448, "shared memory per CTA");
  float4* stage_all = reinterpret_cast<float4*>(smem + STAGES * STAGE_BYTES);   // 8 x 4 KB epilogue staging
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES + kEpiStageBytes);
  uint64_t* empty = full + STAGES;
  uint64_t* acc_full = empty + STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int unit = int(blockIdx.x);
  const int units = int(gridDim.x);
  const int n_tiles = (p.N + BN - 1) / BN, m_tiles = (p.M + BM - 1) / BM;
  const int tiles = n_tiles * m_tiles;
  const int KB = p.KB;
  constexpr uint32_t kCols = 2 * BN < 32 ? 32 : 2 * BN;
  auto tile_n0 = [&](int t) { return (t % n_tiles) * BN; };
  auto tile_m0 = [&](int t) { return (t / n_tiles) * BM; };

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], kPersistThreads - 64);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tmB)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      uint32_t g = 0;
      for (int t = unit; t < tiles && !*abort_flag; t += units) {
        const int n0 = tile_n0(t), m0 = tile_m0(t);
        for (int kb = 0; kb < KB; ++kb, ++g) {
          const int s = g % STAGES;
          if (!mbar_wait(&empty[s], ((g / STAGES) & 1) ^ 1)) {
            atomicExch(p.err, 4);
            *abort_flag = 1;
            break;
          }
          char* sa = smem + s * STAGE_BYTES;
          mbar_expect_tx(&full[s], STAGE_BYTES);
          load_kblock<KIND, BN>(p, kb, m0, n0, sa, sa + A_BYTES, &full[s]);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = instr_desc(BN, KindTraits<KIND>::a_mn, KindTraits<KIND>::b_mn);
      uint32_t g = 0, lt = 0;
      for (int t = unit; t < tiles && !*abort_flag; t += units, ++lt) {
        const uint32_t b = lt & 1;
        // E_TMA: the epilogue warps arrive once per buffer before the first
        // tile, after writing its starting value
        if (!mbar_wait(&acc_empty[b], ((lt >> 1) & 1) ^ ((EPI & E_TMA) ? 0u : 1u))) {
          atomicExch(p.err, 5);
          *abort_flag = 1;
          mbar_expect_tx(&acc_full[b], 0);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + b * BN;
        bool ok = true;
        for (int kb = 0; kb < KB; ++kb, ++g) {
          const int s = g % STAGES;
          if (!mbar_wait(&full[s], (g / STAGES) & 1)) {
            atomicExch(p.err, 6);
            *abort_flag = 1;
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(smem + s * STAGE_BYTES);
          const uint32_t b0 = a0 + A_BYTES;
#pragma unroll
          for (int k = 0; k < BK / UK; ++k) {
            uint64_t ad, bd;
            if (KindTraits<KIND>::a_mn) ad = smem_desc(a0 + k * UK * 128, BK * 128, 1024);
            else ad = smem_desc(a0 + k * UK * 2, 16, 1024);
            if (KindTraits<KIND>::b_mn) bd = smem_desc(b0 + k * UK * 128, BK * 128, 1024);
            else bd = smem_desc(b0 + k * UK * 2, 16, 1024);
            mma_f16(d, ad, bd, idesc, ((EPI & E_TMA) || kb > 0 || k > 0) ? 1u : 0u);
          }
          mma_commit(&empty[s]);
        }
        if (ok) mma_commit(&acc_full[b]);
        else {
          mbar_expect_tx(&acc_full[b], 0);
          break;
        }
      }
    }
  } else if constexpr ((EPI & E_TMA) != 0) {
    // Epilogue through TMA stores: warp w (2..9) owns TMEM lanes
    // 32 * (w % 4) .. +31 and half of the tile's columns; each lane holds
    // one output row.  Two 2 KB staging buffers per warp alternate, each
    // reused once the TMA store that read it two chunks earlier is done.
    const int q = warp % 4, half = (warp - 2) / 4;
    constexpr int CW = BN / 2;
    const uint32_t tq = tmem + (uint32_t(q * 32) << 16) + uint32_t(half * CW);
    const uint32_t stage0 = smem_u32(stage_all) + uint32_t(warp - 2) * 4096u;
    for (int b = 0; b < 2; ++b) {   // the first two tiles' accumulators start from the bias
      const int t = unit + b * units;
      if (t < tiles) tma_preload<EPI, CW>(p, tq + uint32_t(b * BN), tile_m0(t) + q * 32 + lane, tile_n0(t) + half * CW);
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&acc_empty[b]);
    }
    uint32_t lt = 0, sbuf = 0;
    int issued = 0;
    for (int t = unit; t < tiles; t += units, ++lt) {
      const uint32_t b = lt & 1;
      const int n0 = tile_n0(t) + half * CW, m0 = tile_m0(t) + q * 32;
      const bool ready = mbar_wait(&acc_full[b], (lt >> 1) & 1);
      tc_fence_after();
      if (!ready) {
        atomicExch(p.err, 7);
        *abort_flag = 1;
      }
      if (!ready || *abort_flag) break;
      const uint32_t trow = tq + b * BN;
      uint32_t cur[32], nxt[32];
      tmem_ld32_issue(trow, cur);
      tmem_ld32_wait(cur);
#pragma unroll 1
      for (int c = 0; c < CW; c += 32) {
        const bool more = c + 32 < CW;
        if (more) tmem_ld32_issue(trow + uint32_t(c + 32), nxt);
        if (n0 + c < p.N && m0 < p.M) {   // a box past the end of the output has nothing to write
          if constexpr ((EPI & E_GELU) != 0) {
            // both buffers per chunk (pre-activation, GELU); the GELU is
            // computed while the previous chunk's stores read shared memory
            uint32_t hk[16], gk[16];
            gelu_pack32(cur, hk, gk);
            if (issued > 0) {
              if (lane == 0) bulk_wait_read<0>();
              __syncwarp();
            }
            stage_row64(stage0, lane, hk);
            stage_row64(stage0 + 2048u, lane, gk);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&p.tmO, stage0, n0 + c, m0);
              tma_store_2d(&p.tmG, stage0 + 2048u, n0 + c, m0);
            }
            ++issued;
          } else {
            const uint32_t buf = stage0 + sbuf * 2048u;
            if (issued >= 2) {   // buf's previous store is not the newest: at most one may still read
              if (lane == 0) bulk_wait_read<1>();
              __syncwarp();
            }
            tma_chunk32<EPI>(p, buf, lane, m0 + lane, n0 + c, cur);
            __syncwarp();
            if (lane == 0) tma_store_2d(&p.tmO, buf, n0 + c, m0);
            ++issued;
            sbuf ^= 1u;
          }
        }
        if (more) {
          tmem_ld32_wait(nxt);
#pragma unroll
          for (int j = 0; j < 32; ++j) cur[j] = nxt[j];
        }
      }
      // this warp's part of buffer b is drained: start it for the tile two ahead
      const int t2 = t + 2 * units;
      if (t2 < tiles) {
        tma_preload<EPI, CW>(p, trow, tile_m0(t2) + q * 32 + lane, tile_n0(t2) + half * CW);
        tmem_st_wait();
      }
      tc_fence_before();
      mbar_arrive(&acc_empty[b]);
    }
    if (lane == 0) bulk_wait_all();   // the stores have read shared memory and reached global memory
    __syncwarp();
  } else {
    // Epilogue: warp w (2..9) reads TMEM lanes 32 * (w % 4) .. +31; the two
    // warps of a lane quarter split the tile's columns.
    const int q = warp % 4, half = (warp - 2) / 4;
    constexpr int CW = BN / 2;  // columns per epilogue warp (a multiple of 32)
    uint32_t lt = 0;
    for (int t = unit; t < tiles; t += units, ++lt) {
      const uint32_t b = lt & 1;
      const int n0 = tile_n0(t), m0 = tile_m0(t);
      float bnext[8];
      load_bias8<EPI>(p, lane, n0 + half * CW, bnext);   // in flight during the wait
      const bool ready = mbar_wait(&acc_full[b], (lt >> 1) & 1);
      tc_fence_after();
      if (!ready) {
        atomicExch(p.err, 7);
        *abort_flag = 1;
      }
      if (!ready || *abort_flag) break;
      const uint32_t stage = smem_u32(stage_all) + uint32_t(warp - 2) * 4096u;
      const uint32_t trow = tmem + b * BN + (uint32_t(q * 32) << 16);
      // Software-pipelined: the TMEM load of chunk c + 32 is in flight while
      // chunk c is staged and stored.  Not unrolled: the epilogue runs once
      // per tile from a cold instruction cache, so compact code matters more
      // than loop overhead.
      uint32_t cur[32], nxt[32];
      tmem_ld32_issue(trow + uint32_t(half * CW), cur);
      tmem_ld32_wait(cur);
#pragma unroll 1
      for (int c = half * CW; c < (half + 1) * CW; c += 32) {
        const bool more = c + 32 < (half + 1) * CW;
        float bcur[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) bcur[j] = bnext[j];
        if (more) {
          load_bias8<EPI>(p, lane, n0 + c + 32, bnext);
          tmem_ld32_issue(trow + uint32_t(c + 32), nxt);
        }
        epilogue_chunk32<EPI>(p, stage, lane, m0 + q * 32, n0 + c, cur, bcur);
        if (more) {
          tmem_ld32_wait(nxt);
#pragma unroll
          for (int j = 0; j < 32; ++j) cur[j] = nxt[j];
        }
      }
      tc_fence_before();
      mbar_arrive(&acc_empty[b]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kCols) : "memory");
  }
}

// Pipeline depth.  A stage's round trip (TMA load, MMAs, release) takes
// ~1.5-2.5 us, so the main loop of a narrow tile runs at stages / round trip
// and every stage that fits counts.  The persistent kernel keeps 32 KB of
// epilogue staging; the split-K kernel takes all the rest of the 227 KB.
constexpr int kSmemMax = 232448;
constexpr int stages_of(int bn, bool cluster) {
  const int stage = BM * BK * 2 + bn * BK * 2;
  const int budget = cluster ? kSmemMax - 1024 - 256 - 4 * bn : kSmemBudget;
  return budget / stage > 8 ? 8 : budget / stage;
}
template <int KIND, int BN, bool CLUSTER>
constexpr int stages_for() {
  return stages_of(BN, CLUSTER);
}
inline size_t pipeline_bytes(int bn) {   // the split-K kernel's pipeline buffers
  return size_t(stages_of(bn, true)) * (BM * BK * 2 + bn * BK * 2);
}
template <int KIND, int BN>
constexpr size_t smem_bytes(bool cluster) {
  return size_t(stages_of(BN, cluster)) * (BM * BK * 2 + BN * BK * 2) + 1024 + 256 +
         (cluster ? 4 * BN : kEpiStageBytes);
}

// The kernel of (KIND, BN, EPI), split-K (cluster) or persistent, with its
// dynamic shared memory; instantiated in the translation unit of its kind
// group (k_tc_gemm_fwd.cu, k_tc_gemm_dgrad.cu, k_tc_gemm_wgrad.cu).
template <int KIND, int BN, int EPI>
KernelFn kernel_of(bool cluster, size_t* smem) {
  *smem = smem_bytes<KIND, BN>(cluster);
  if constexpr ((EPI & E_TMA) != 0) {   // the persistent kernel only
    if (cluster) return nullptr;
    return tc_gemm_persistent<KIND, BN, stages_for<KIND, BN, false>(), EPI>;
  } else {
    if (cluster) return tc_gemm_kernel<KIND, BN, stages_for<KIND, BN, true>(), EPI>;
    return tc_gemm_persistent<KIND, BN, stages_for<KIND, BN, false>(), EPI>;
  }
}
template <int KIND, int EPI>
KernelFn kernel_bn(int bn, bool cluster, size_t* smem) {
  if (bn == 256) return kernel_of<KIND, 256, EPI>(cluster, smem);
  if (bn == 128) return kernel_of<KIND, 128, EPI>(cluster, smem);
  if (bn == 64) return kernel_of<KIND, 64, EPI>(cluster, smem);
  return nullptr;
}

// The kernel of (kind, bn, epi) with its shared memory, or nullptr for a
// combination no planner asks for; one per kind group and translation unit.
KernelFn pick_fwd(int kind, int bn, bool cluster, int epi, size_t* smem);     // LIN_FWD, CONV_FPROP
KernelFn pick_dgrad(int kind, int bn, bool cluster, int epi, size_t* smem);   // LIN_DGRAD, CONV_DGRAD
KernelFn pick_wgrad(int kind, int bn, bool cluster, int epi, size_t* smem);   // LIN_WGRAD, CONV_WGRAD

}  // namespace tcg
}  // namespace fo
