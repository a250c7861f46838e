// Tensor-core GEMM / implicit-GEMM convolution for sm_103a: tcgen05.mma
// (kind::f16, bf16 operands, fp32 accumulator in TMEM) fed by TMA tiles in
// 128-byte-swizzled shared memory, with a warp-specialised pipeline:
//   warp 0      TMA producer (one thread)
//   warp 1      TMEM allocator and MMA issuer (one thread)
//   warps 2..5  epilogue: tcgen05.ld of the 128 x BN accumulator, then the
//               bias / ReLU / bf16 or fp32 store (or an fp32 split-K partial)
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
#include "fo_server_impl.h"
#include "fo_ptx.cuh"
#include "fo_tc.h"

#include <cuda.h>
#include <algorithm>
#include <cstring>
#include <map>
#include <vector>

namespace fo {

namespace {

enum Kind { LIN_FWD = 0, LIN_DGRAD = 1, LIN_WGRAD = 2, CONV_FPROP = 3, CONV_DGRAD = 4, CONV_WGRAD = 5 };

constexpr int BM = 128;      // UMMA M (cta_group::1)
constexpr int BK = 64;       // k-block: one 128-byte swizzle row of bf16
constexpr int UK = 16;       // UMMA K for kind::f16
constexpr int kThreads = 192;
constexpr int kSmemBudget = 200 * 1024;

struct TcParams {
  CUtensorMap tmA;
  CUtensorMap tmB;
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

// Epilogue of 32 consecutive outputs (m, n..n+31) held by one thread: bias,
// ReLU, ReLU mask, accumulate, store as fp32 or bf16 (16-byte accesses).
// `sbias`: shared-memory address of the bias values for columns n..n+31.
// Columns >= N (the ragged last tile; N is a multiple of 8) are not touched.
// bf16 outputs take their ReLU-mask and accumulate operands preloaded by
// load_row32 (so that a caller can fetch them ahead of time).
__device__ __forceinline__ void load_row32(const TcParams& p, int m_gemm, int n, uint4 (&mk)[4], uint4 (&ac)[4]) {
  const int nv = p.N - n;
  if (p.out_f32 || nv <= 0 || m_gemm >= p.M) return;
  const size_t m = out_row(p, m_gemm);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (8 * j >= nv) break;
    if (p.mask) mk[j] = *reinterpret_cast<const uint4*>(p.mask + m * p.ldo + n + 8 * j);
    if (p.acc) ac[j] = *reinterpret_cast<const uint4*>(reinterpret_cast<const bf16*>(p.out) + m * p.ldo + n + 8 * j);
  }
}
__device__ __forceinline__ void store_row32(const TcParams& p, int m_gemm, int n, float (&v)[32], uint32_t sbias,
                                            const uint4 (&mk)[4], const uint4 (&ac)[4]) {
  const size_t m = out_row(p, m_gemm);
  const int nv = p.N - n;   // valid columns from n
  if (nv <= 0) return;
  if (p.bias) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 b = ld_shared4(sbias + 16u * j);
      v[4 * j] += b.x; v[4 * j + 1] += b.y; v[4 * j + 2] += b.z; v[4 * j + 3] += b.w;
    }
  }
  if (p.relu)
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = fmaxf(v[j], 0.f);
  if (p.out_f32) {
    if (p.mask) {
      const uint4* mkp = reinterpret_cast<const uint4*>(p.mask + m * p.ldo + n);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (8 * j >= nv) break;
        const uint4 u = mkp[j];
        const bf16* e = reinterpret_cast<const bf16*>(&u);
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (!(__bfloat162float(e[q]) > 0.f)) v[8 * j + q] = 0.f;
      }
    }
    float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(p.out) + m * p.ldo + n);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (4 * j >= nv) break;
      if (p.acc) {
        const float4 o = dst[j];
        v[4 * j] += o.x; v[4 * j + 1] += o.y; v[4 * j + 2] += o.z; v[4 * j + 3] += o.w;
      }
      dst[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
    }
  } else {
    uint4* dst = reinterpret_cast<uint4*>(reinterpret_cast<bf16*>(p.out) + m * p.ldo + n);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (8 * j >= nv) break;
      if (p.mask) {
        const bf16* e = reinterpret_cast<const bf16*>(&mk[j]);
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (!(__bfloat162float(e[q]) > 0.f)) v[8 * j + q] = 0.f;
      }
      if (p.acc) {
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

// Coalesced epilogue of a 32-row x 32-column accumulator chunk held one row
// per lane (lane = row, r[j] = column j).  The warp stages the chunk in its
// 4 KB shared-memory buffer (16-byte units XOR-swizzled by row, so both the
// row-wise writes and the column-wise reads are free of bank conflicts), then
// reads it back so that consecutive lanes own consecutive columns of a row:
// bias, ReLU, ReLU mask, accumulate and the stores then touch whole 32-byte
// sectors (bf16: 8 rows x 64 B per instruction; fp32: 4 rows x 128 B).
// The bias values lane `lane` applies in epilogue_chunk32 for the chunk at
// column n: 8 columns from 8 * (lane % 4) for bf16 outputs, 4 columns from
// 4 * (lane % 8) for fp32 outputs (zeros without a bias).
__device__ __forceinline__ void load_bias8(const TcParams& p, int lane, int n, float (&b)[8]) {
  float4 b0 = make_float4(0.f, 0.f, 0.f, 0.f), b1 = b0;
  if (p.bias && n + (p.out_f32 ? 4 * (lane & 7) : 8 * (lane & 3)) < p.N) {
    const float4* src = reinterpret_cast<const float4*>(p.bias + n);
    if (p.out_f32) {
      b0 = __ldg(src + (lane & 7));
    } else {
      b0 = __ldg(src + 2 * (lane & 3));
      b1 = __ldg(src + 2 * (lane & 3) + 1);
    }
  }
  b[0] = b0.x; b[1] = b0.y; b[2] = b0.z; b[3] = b0.w; b[4] = b1.x; b[5] = b1.y; b[6] = b1.z; b[7] = b1.w;
}

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
  if (!p.out_f32) {
#pragma unroll
    for (int it = 0; it < 4; ++it) {
      const int mg = m_base + it * 8 + (lane >> 2);
      ok[it] = mg < p.M && n + 8 * co < p.N;
      off[it] = ok[it] ? out_row(p, mg) * p.ldo + n + 8 * co : 0;
      if (p.mask && ok[it]) mk[it] = *reinterpret_cast<const uint4*>(p.mask + off[it]);
      if (p.acc && ok[it]) ac[it] = *reinterpret_cast<const uint4*>(reinterpret_cast<const bf16*>(p.out) + off[it]);
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j)
    st_shared4(stage + 16u * (lane * 8 + (j ^ (lane & 7))), r[4 * j], r[4 * j + 1], r[4 * j + 2], r[4 * j + 3]);
  __syncwarp();
  if (p.out_f32) {
    const int cq = lane & 7;                 // 16-byte unit: columns 4cq .. 4cq+3
#pragma unroll 1
    for (int it = 0; it < 8; ++it) {
      const int rr = it * 4 + (lane >> 3);
      const int mg = m_base + rr;
      const float4 v = ld_shared4(stage + 16u * (rr * 8 + (cq ^ (rr & 7))));
      if (mg < p.M && n + 4 * cq < p.N) {
        const size_t m = out_row(p, mg);
        float e[4] = {v.x + b[0], v.y + b[1], v.z + b[2], v.w + b[3]};
        if (p.relu)
#pragma unroll
          for (int q = 0; q < 4; ++q) e[q] = fmaxf(e[q], 0.f);
        if (p.mask) {
          const uint2 u = *reinterpret_cast<const uint2*>(p.mask + m * p.ldo + n + 4 * cq);
          const bf16* mkp = reinterpret_cast<const bf16*>(&u);
#pragma unroll
          for (int q = 0; q < 4; ++q)
            if (!(__bfloat162float(mkp[q]) > 0.f)) e[q] = 0.f;
        }
        float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(p.out) + m * p.ldo + n) + cq;
        if (p.acc) {
          const float4 o = *dst;
          e[0] += o.x; e[1] += o.y; e[2] += o.z; e[3] += o.w;
        }
        *dst = make_float4(e[0], e[1], e[2], e[3]);
      }
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
        if (p.relu)
#pragma unroll
          for (int q = 0; q < 8; ++q) e[q] = fmaxf(e[q], 0.f);
        if (p.mask) {
          const bf16* mkp = reinterpret_cast<const bf16*>(&mk[it]);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (!(__bfloat162float(mkp[q]) > 0.f)) e[q] = 0.f;
        }
        if (p.acc) {
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
  } else if (p.chunk_b) {  // CONV_WGRAD, all chunks of the tile in one box
    const int tap = n0 / p.ntap_ch, ci0 = n0 % p.ntap_ch;
    const int r = tap / p.ksz, s = tap % p.ksz;
    const int pix0 = kb * BK;
    const int n_img = pix0 / HW, h0 = (pix0 % HW) / p.W;
    tma_5d(sb, &p.tmB, bar, 0, s - p.pad, h0 * p.stride + r - p.pad, n_img, ci0 / 64);
  } else {  // CONV_WGRAD: N index = tap * Ci + ci; K = output pixel
    const int tap = n0 / p.ntap_ch, ci0 = n0 % p.ntap_ch;
    const int r = tap / p.ksz, s = tap % p.ksz;
    const int pix0 = kb * BK;
    const int n_img = pix0 / HW, h0 = (pix0 % HW) / p.W;   // H, W: output grid
#pragma unroll
    for (int j = 0; j < BN / 64; ++j)
      tma_4d(sb + j * BK * 128, &p.tmB, bar, ci0 + j * 64, s - p.pad, h0 * p.stride + r - p.pad, n_img);
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
template <int KIND, int BN, int STAGES>
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
    load_row32(p, mg, n0 + 32 * c0, mk, ac);
    if (!mbar_wait(rbar, 0)) atomicExch(p.err, 9);
#pragma unroll 1
    for (int c = c0; c < c1; ++c) {
      if (c + 1 < c1) load_row32(p, mg, n0 + 32 * (c + 1), mk2, ac2);
      uint32_t r[32];
      tmem_ld32(trow + uint32_t(32 * c), r);
      if (mg < p.M) {
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
        store_row32(p, mg, n0 + 32 * c, v, smem_u32(sbias) + uint32_t(32 * c) * 4u, mk, ac);
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
template <int KIND, int BN, int STAGES>
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
        if (!mbar_wait(&acc_empty[b], ((lt >> 1) & 1) ^ 1)) {
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
            mma_f16(d, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
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
      load_bias8(p, lane, n0 + half * CW, bnext);   // in flight during the wait
      const bool ready = mbar_wait(&acc_full[b], (lt >> 1) & 1);
      tc_fence_after();
      if (!ready) {
        atomicExch(p.err, 7);
        *abort_flag = 1;
      }
      if (!ready || *abort_flag) break;
      const uint32_t stage = smem_u32(stage_all) + uint32_t(warp - 2) * 4096u;
      // Not unrolled: the epilogue runs once per tile from a cold instruction
      // cache, so compact code matters more than loop overhead.
#pragma unroll 1
      for (int c = half * CW; c < (half + 1) * CW; c += 32) {
        float bcur[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) bcur[j] = bnext[j];
        if (c + 32 < (half + 1) * CW) load_bias8(p, lane, n0 + c + 32, bnext);
        uint32_t r[32];
        tmem_ld32(tmem + b * BN + (uint32_t(q * 32) << 16) + uint32_t(c), r);
        epilogue_chunk32(p, stage, lane, m0 + q * 32, n0 + c, r, bcur);
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

typedef void (*KernelFn)(const TcParams);

template <int KIND, int BN>
KernelFn kernel_ptr(bool cluster) {
  if (cluster) return tc_gemm_kernel<KIND, BN, stages_for<KIND, BN, true>()>;
  return tc_gemm_persistent<KIND, BN, stages_for<KIND, BN, false>()>;
}

KernelFn pick_kernel(int kind, int bn, bool cluster, size_t* smem) {
#define FO_PICK(K)                                                  \
  if (kind == K) {                                                  \
    if (bn == 256) { *smem = smem_bytes<K, 256>(cluster); return kernel_ptr<K, 256>(cluster); } \
    if (bn == 128) { *smem = smem_bytes<K, 128>(cluster); return kernel_ptr<K, 128>(cluster); } \
    *smem = smem_bytes<K, 64>(cluster);                                    \
    return kernel_ptr<K, 64>(cluster);                               \
  }
  FO_PICK(LIN_FWD)
  FO_PICK(LIN_DGRAD)
  FO_PICK(LIN_WGRAD)
  FO_PICK(CONV_FPROP)
  FO_PICK(CONV_DGRAD)
  FO_PICK(CONV_WGRAD)
#undef FO_PICK
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
              const uint32_t* box, const uint32_t* elem = nullptr) {
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
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
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
  bool input_A = false;   // operand fed by the uploaded batch (tensor 0)
  bool input_B = false;
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
int active_clusters(TcContext* c, int kind, int bn, int S) {
  const int key = (kind * 512 + bn) * 16 + S;
  auto it = c->cluster_fit.find(key);
  if (it != c->cluster_fit.end()) return it->second;
  size_t smem = 0;
  KernelFn fn = pick_kernel(kind, bn, true, &smem);
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
//    so 256-wide tiles run at ~3/4 of the MMA peak and 128-wide ones at
//    ~3/8: the floor above;
//  * a CTA pays a start-up ramp and the epilogue of its last tile (earlier
//    epilogues overlap the next tile's MMAs), a K-split cluster pays the
//    staging and distributed-shared-memory reduction of its partial tiles,
//    and clusters run in waves of what the occupancy calculator fits at once.
// Candidate widths divide `ndiv` (N, or the channels of one tap for the
// weight gradient, whose N index runs over taps x channels).
void choose_tiles(TcContext* c, TcGemm* g, int M, int N, int KB, int ndiv) {
  const bool win_a = g->kind == CONV_FPROP || g->kind == CONV_DGRAD;
  const bool win_b = g->kind == CONV_WGRAD;
  double best = 1e30;
  int best_bn = 0, best_s = 1;
  for (int bn : {256, 128, 64}) {
    // window kinds tile whole taps; the plain GEMMs take a ragged last tile
    if ((win_a || win_b) && (ndiv % bn || N % bn)) continue;
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
        const int fit = active_clusters(c, g->kind, bn, splits);
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
  g->p.M = M;
  g->p.N = N;
  g->flops = 2.0 * M * N * K;
  g->p.err = c->err;
  g->fn = pick_kernel(g->kind, g->bn, g->splits > 1, &g->smem);
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

TcGemm* tc_plan_forward(TcContext* c, fo_server* s, int i, void* out, bool relu) {
  if (!c || !bf16_server(s) || getenv("FO_NO_TC")) return nullptr;
  const fo_op& op = s->ops[i];
  const Tensor& a = s->T[op.in0];
  const Tensor& o = s->T[i + 1];
  if (o.dt != kBF16) return nullptr;  // fp32 logits: CUDA-core path
  TcGemm* g = new TcGemm();
  g->p.out = out;
  g->p.ldo = o.C;
  g->p.relu = relu ? 1 : 0;
  g->p.bias = op.bias ? s->theta + s->segs[s->op_segs[i][1]].off : nullptr;
  const bf16* w = s->shadow + s->segs[s->op_segs[i][0]].off;
  if (plain_gemm(op)) {
    if (!plain_gemm_ok(op)) { delete g; return nullptr; }
    g->kind = LIN_FWD;
    g->name = op.kind == FO_OP_LINEAR ? "tc_linear_fwd" : "tc_conv1x1_fwd";
    int M = int(a.rows()), KB = (op.cin + 63) / 64;
    choose_tiles(c, g, M, op.cout, KB, op.cout);
    const int bn = g->bn;
    g->input_A = (op.in0 == 0);
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
  g->input_A = (op.in0 == 0);
  if (g->input_A) {
    g->slot_maps.resize(s->cfg.omega);
    for (int sl = 0; sl < s->cfg.omega; ++sl)
      if (!map_window(&g->slot_maps[sl], s->slab + size_t(sl) * s->slot_stride, a.N, a.H, a.W, a.C, Wo, box_rows, box_imgs, st)) { delete g; return nullptr; }
  } else if (!map_window(&g->p.tmA, tensor_act(s, op.in0), a.N, a.H, a.W, a.C, Wo, box_rows, box_imgs, st)) { delete g; return nullptr; }
  if (!map_2d(&g->p.tmB, w, op.cout, int64_t(g->p.taps) * op.cin, bn)) { delete g; return nullptr; }
  return finish(c, g, M, op.cout, double(g->p.taps) * op.cin);
}

bool tc_plan_dgrad(TcContext* c, fo_server* s, int i, int accumulate, void* dx, const void* mask,
                   std::vector<TcGemm*>* out, bool* zero_first) {
  out->clear();
  *zero_first = false;
  if (!c || !bf16_server(s) || getenv("FO_NO_TC")) return false;
  const fo_op& op = s->ops[i];
  const Tensor& a = s->T[op.in0];
  const Tensor& o = s->T[i + 1];
  if (o.dt != kBF16) return false;
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
    g->input_B = (op.in0 == 0);
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
  g->input_B = (op.in0 == 0);
  if (!map_2d(&g->p.tmA, o.grad, P, op.cout, BK)) { delete g; return nullptr; }
  CUtensorMap ca;
  if (map_chunked(&ca, o.grad, P, op.cout, BK, BM / 64)) { g->p.tmA = ca; g->p.chunk_a = 1; }
  const int nchunk = g->bn / 64;
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
