// Tensor-core multi-head attention for sequences of up to 128 tokens and
// head width 64 (bf16 activations): one CTA per (sequence, head), the whole
// 128 x 128 score tile in TMEM.  Same operation as the CUDA-core kernels
// (scaled dot-product attention with keys j >= length[b] masked out):
//   forward   S = Q K^T (TMEM) -> row maximum M of S / sqrt(64) -> P~ =
//             exp(S / 8 - M) (bf16, shared memory) and its row sum ->
//             O = P~ V (TMEM) -> O / row sum (bf16), plus the row
//             log-sum-exp of the scaled scores for the backward pass;
//   backward  S = Q K^T and dP = dO V^T (TMEM) -> P = exp(S / 8 - lse),
//             dS = P (dP - rowsum(dO * O)) / 8 (bf16, shared memory) ->
//             dV = P^T dO, dQ = dS K, dK = dS^T Q (TMEM) -> d(q|k|v).
// Operand tiles are 128 rows x 64 bf16 (128-byte rows, 128-byte swizzle),
// loaded by TMA from the packed q|k|v [B*L, 3C] and dO [B*L, C] (the
// backward reads O's rows directly for rowsum(dO * O));
// P (P~ in the forward) and dS are written by the softmax threads in the same swizzled layout as
// two 64-column sub-tiles, which serves both as a K-major operand (P V,
// dS K) and as an MN-major one (P^T dO, dS^T Q).
// Warp roles: warp 0 issues the TMA loads, warp 1 owns TMEM and issues the
// MMAs (one thread each), warps 2..9 do the softmax and the stores: warp w
// reads TMEM lane quarter w % 4 (32 rows) and takes keys 64 * ((w - 2) / 4)
// .. +63 of them, so every row is shared by two threads (the forward pass
// combines their partial maxima and sums through shared memory).  Waits are
// bounded (error word 11..16).
#include "fo_common.cuh"
#include "fo_kernels.h"
#include "fo_ptx.cuh"
#include "fo_tc.h"

namespace fo {

namespace {

constexpr int kAttnThreads = 320;
constexpr int kSoftmaxThreads = 256;      // warps 2..9
constexpr int kTile = 16384;              // 128 rows x 64 bf16
constexpr float kScale = 0.125f;          // 1 / sqrt(64)

struct AttnParams {
  CUtensorMap tm_qkv;     // [B*L, 3C], box 64 x 128
  CUtensorMap tm_do;      // [B*L, C],  box 64 x 128 (backward)
  const int32_t* len;     // [B]
  const bf16* o;          // backward: the forward output O [B*L, C] (for rowsum(dO * O))
  bf16* out;              // forward: O [B*L, C]; backward: d(q|k|v) [B*L, 3C]
  float* lse;             // [B * heads * L]
  int L, C, heads, acc;
  int* err;
};

// Byte offset of 16-byte unit u (0..7) of row r in a 128-byte-swizzled
// 128 x 64 bf16 tile (8-row groups of 1024 bytes, units XOR-permuted by row).
__device__ __forceinline__ uint32_t sw_off(int r, int u) {
  return uint32_t((r >> 3) * 1024 + (r & 7) * 128 + ((u ^ (r & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ char* align1024(char* p) {
  return reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// 32 accumulator columns of this lane's row -> 32 bf16 at dst (optionally
// added to what is there).
__device__ __forceinline__ void store_row32(bf16* dst, const uint32_t (&r)[32], bool acc) {
  uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    float v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = __uint_as_float(r[8 * q + e]);
    if (acc) {
      const uint4 o = d4[q];
      const bf16* ob = reinterpret_cast<const bf16*>(&o);
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] += __bfloat162float(ob[e]);
    }
    d4[q] = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                       pack_bf16x2(v[6], v[7]));
  }
}

__global__ void __launch_bounds__(kAttnThreads, 1) attn_fwd_tc_k(const __grid_constant__ AttnParams p) {
  extern __shared__ __align__(1024) char smem_raw[];
  char* sm = align1024(smem_raw);
  char* sQ = sm;
  char* sK = sm + kTile;
  char* sV = sm + 2 * kTile;
  char* sP = sm + 3 * kTile;                       // two sub-tiles (keys 0..63, 64..127)
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + 5 * kTile);   // ld, s, p, o
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 4);
  float2* xch = reinterpret_cast<float2*>(sm + 5 * kTile + 64);   // [half][row]: partial maxima, then sums

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int bh = blockIdx.x, b = bh / p.heads, h = bh % p.heads;
  const int row0 = b * p.L;
  if (threadIdx.x == 0) {
    mbar_init(&bars[0], 1);
    mbar_init(&bars[1], 1);
    mbar_init(&bars[2], kSoftmaxThreads);
    mbar_init(&bars[3], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tm_qkv)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tslot)),
                 "r"(256)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;          // S: columns 0..127, O: 128..191
  pdl_trigger();   // this block holds its tensor memory
  pdl_wait();      // the previous kernel's writes are visible from here on

  if (warp == 0) {
    if (lane == 0) {
      mbar_expect_tx(&bars[0], 3 * kTile);
      tma_2d(sQ, &p.tm_qkv, &bars[0], h * 64, row0);
      tma_2d(sK, &p.tm_qkv, &bars[0], p.C + h * 64, row0);
      tma_2d(sV, &p.tm_qkv, &bars[0], 2 * p.C + h * 64, row0);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      if (!mbar_wait(&bars[0], 0)) atomicExch(p.err, 11);
      tc_fence_after();
      constexpr uint32_t id_s = instr_desc(128, false, false);
#pragma unroll
      for (int k = 0; k < 4; ++k)
        mma_f16(tmem, smem_desc(smem_u32(sQ) + 32 * k, 16, 1024), smem_desc(smem_u32(sK) + 32 * k, 16, 1024), id_s,
                k > 0 ? 1u : 0u);
      mma_commit(&bars[1]);
      if (!mbar_wait(&bars[2], 0)) atomicExch(p.err, 12);
      tc_fence_after();
      constexpr uint32_t id_o = instr_desc(64, false, true);
#pragma unroll
      for (int k = 0; k < 8; ++k)
        mma_f16(tmem + 128, smem_desc(smem_u32(sP) + (k >> 2) * kTile + 32 * (k & 3), 16, 1024),
                smem_desc(smem_u32(sV) + 2048 * k, kTile, 1024), id_o, k > 0 ? 1u : 0u);
      mma_commit(&bars[3]);
    }
  } else {
    const int q = warp % 4, i = q * 32 + lane, hf = (warp - 2) / 4;
    const uint32_t trow = tmem + (uint32_t(q * 32) << 16) + uint32_t(64 * hf);   // this thread's 64 keys
    const int n = min(p.len[b], p.L);
    if (!mbar_wait(&bars[1], 0)) atomicExch(p.err, 13);
    tc_fence_after();
    // the row maximum over this thread's keys, combined with the other half
    uint32_t r[32];
    float m = -INFINITY;
#pragma unroll 1
    for (int c = 0; c < 2; ++c) {
      tmem_ld32(trow + 32 * c, r);
      const int j0 = 64 * hf + 32 * c;
#pragma unroll
      for (int e = 0; e < 32; ++e)
        if (j0 + e < n) m = fmaxf(m, __uint_as_float(r[e]) * kScale);
    }
    xch[hf * 128 + i] = make_float2(m, 0.f);
    asm volatile("bar.sync 1, %0;" ::"n"(kSoftmaxThreads) : "memory");
    const float M = fmaxf(m, xch[(1 - hf) * 128 + i].x);
    // P~ = exp(s / 8 - M) (bf16, unnormalised: one exponential per score) and
    // its row sum; O = P~ V is normalised by the sum in the store below
    float sum = 0.f;
    const uint32_t p_base = smem_u32(sP) + uint32_t(hf) * kTile;
#pragma unroll 1
    for (int c = 0; c < 2; ++c) {
      tmem_ld32(trow + 32 * c, r);
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        float v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const int j = 64 * hf + 32 * c + 8 * g + e;
          v[e] = j < n ? __expf(__uint_as_float(r[8 * g + e]) * kScale - M) : 0.f;
          sum += v[e];
        }
        st_shared4(p_base + sw_off(i, c * 4 + g), pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                   pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
      }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // P~ visible to the tensor cores
    tc_fence_before();
    mbar_arrive(&bars[2]);
    // the row sum over both halves, while the tensor cores form O
    xch[256 + hf * 128 + i] = make_float2(sum, 0.f);
    asm volatile("bar.sync 1, %0;" ::"n"(kSoftmaxThreads) : "memory");
    const float S = sum + xch[256 + (1 - hf) * 128 + i].x;
    const float inv = S > 0.f ? 1.f / S : 0.f;
    if (hf == 0 && i < p.L) p.lse[size_t(bh) * p.L + i] = M + logf(S);
    if (!mbar_wait(&bars[3], 0)) atomicExch(p.err, 14);
    tc_fence_after();
    // O: 64 columns at TMEM column 128; each half of the pair stores 32
    tmem_ld32(tmem + (uint32_t(q * 32) << 16) + 128 + 32 * hf, r);
#pragma unroll
    for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * inv);
    if (i < p.L) store_row32(p.out + size_t(row0 + i) * p.C + h * 64 + 32 * hf, r, false);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256) : "memory");
  }
}

// Two CTAs per SM: 7 tiles of shared memory (112 KB) and 256 TMEM columns.
// V is read only by the first MMA phase, so P's first sub-tile takes its
// buffer once that phase has completed; O is read from global memory (only
// its row sums with dO are needed); dQ, dV and dK take the TMEM columns of S
// and dP, which the softmax warps have read before the second phase starts.
__global__ void __launch_bounds__(kAttnThreads, 2) attn_bwd_tc_k(const __grid_constant__ AttnParams p) {
  extern __shared__ __align__(1024) char smem_raw[];
  char* sm = align1024(smem_raw);
  char* sQ = sm;
  char* sK = sm + kTile;
  char* sV = sm + 2 * kTile;
  char* sP = sm + 2 * kTile;      // two sub-tiles: V's buffer after the first phase, then the next
  char* sdO = sm + 4 * kTile;
  char* sdS = sm + 5 * kTile;     // two sub-tiles
  // barriers (ld, s, p, g) and the TMEM slot: in the alignment slack below
  // the tiles when it has room, else after them (the request covers both)
  const bool low = sm - smem_raw >= 64;
  uint64_t* bars = reinterpret_cast<uint64_t*>(low ? smem_raw : sm + 7 * kTile);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 4);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int bh = blockIdx.x, b = bh / p.heads, h = bh % p.heads;
  const int row0 = b * p.L;
  if (threadIdx.x == 0) {
    mbar_init(&bars[0], 1);
    mbar_init(&bars[1], 1);
    mbar_init(&bars[2], kSoftmaxThreads);
    mbar_init(&bars[3], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tm_qkv)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&p.tm_do)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tslot)),
                 "r"(256)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // TMEM columns: S 0..127 and dP 128..255; then dQ 0..63, dV 128..191, dK 192..255
  const uint32_t tmem = *tslot;
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      mbar_expect_tx(&bars[0], 4 * kTile);
      tma_2d(sQ, &p.tm_qkv, &bars[0], h * 64, row0);
      tma_2d(sK, &p.tm_qkv, &bars[0], p.C + h * 64, row0);
      tma_2d(sV, &p.tm_qkv, &bars[0], 2 * p.C + h * 64, row0);
      tma_2d(sdO, &p.tm_do, &bars[0], h * 64, row0);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      if (!mbar_wait(&bars[0], 0)) atomicExch(p.err, 15);
      tc_fence_after();
      constexpr uint32_t id_nn128 = instr_desc(128, false, false);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        mma_f16(tmem, smem_desc(smem_u32(sQ) + 32 * k, 16, 1024), smem_desc(smem_u32(sK) + 32 * k, 16, 1024),
                id_nn128, k > 0 ? 1u : 0u);
        mma_f16(tmem + 128, smem_desc(smem_u32(sdO) + 32 * k, 16, 1024),
                smem_desc(smem_u32(sV) + 32 * k, 16, 1024), id_nn128, k > 0 ? 1u : 0u);
      }
      mma_commit(&bars[1]);
      if (!mbar_wait(&bars[2], 0)) atomicExch(p.err, 16);
      tc_fence_after();
      constexpr uint32_t id_tt = instr_desc(64, true, true);    // dV, dK: A and B MN-major
      constexpr uint32_t id_nt = instr_desc(64, false, true);   // dQ: A K-major, B MN-major
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const uint32_t acc = k > 0 ? 1u : 0u;
        // dV[j][d] = sum_i P[i][j] dO[i][d]
        mma_f16(tmem + 128, smem_desc(smem_u32(sP) + 2048 * k, kTile, 1024),
                smem_desc(smem_u32(sdO) + 2048 * k, kTile, 1024), id_tt, acc);
        // dQ[i][d] = sum_j dS[i][j] K[j][d]
        mma_f16(tmem, smem_desc(smem_u32(sdS) + (k >> 2) * kTile + 32 * (k & 3), 16, 1024),
                smem_desc(smem_u32(sK) + 2048 * k, kTile, 1024), id_nt, acc);
        // dK[j][d] = sum_i dS[i][j] Q[i][d]
        mma_f16(tmem + 192, smem_desc(smem_u32(sdS) + 2048 * k, kTile, 1024),
                smem_desc(smem_u32(sQ) + 2048 * k, kTile, 1024), id_tt, acc);
      }
      mma_commit(&bars[3]);
    }
  } else {
    const int q = warp % 4, i = q * 32 + lane, hf = (warp - 2) / 4;   // keys 64 hf .. +63
    const uint32_t trow = tmem + (uint32_t(q * 32) << 16);
    const int n = min(p.len[b], p.L);
    const bool live = i < p.L;          // rows past the sequence get P = dS = 0
    // D_i = sum_d dO[i][d] O[i][d]: O's row from global memory (in flight
    // during the TMA wait), dO's from the swizzled tile
    uint4 orow[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) orow[u] = make_uint4(0u, 0u, 0u, 0u);
    if (live) {
      const uint4* src = reinterpret_cast<const uint4*>(p.o + size_t(row0 + i) * p.C + h * 64);
#pragma unroll
      for (int u = 0; u < 8; ++u) orow[u] = src[u];
    }
    if (!mbar_wait(&bars[0], 0)) atomicExch(p.err, 15);
    float D = 0.f;
    const uint32_t do_base = smem_u32(sdO);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const float4 a = ld_shared4(do_base + sw_off(i, u));
      const bf16* ab = reinterpret_cast<const bf16*>(&a);
      const bf16* cb = reinterpret_cast<const bf16*>(&orow[u]);
#pragma unroll
      for (int e = 0; e < 8; ++e) D = fmaf(__bfloat162float(ab[e]), __bfloat162float(cb[e]), D);
    }
    const float lse = live ? p.lse[size_t(bh) * p.L + i] : 0.f;
    if (!mbar_wait(&bars[1], 0)) atomicExch(p.err, 13);
    tc_fence_after();
    const uint32_t p_base = smem_u32(sP), ds_base = smem_u32(sdS);
#pragma unroll 1
    for (int c = 2 * hf; c < 2 * hf + 2; ++c) {
      uint32_t rs[32], rp[32];
      tmem_ld32(trow + 32 * c, rs);
      tmem_ld32(trow + 128 + 32 * c, rp);
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        float pv[8], dv[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const int j = 32 * c + 8 * g + e;
          const float pj = (live && j < n) ? __expf(__uint_as_float(rs[8 * g + e]) * kScale - lse) : 0.f;
          pv[e] = pj;
          dv[e] = pj * (__uint_as_float(rp[8 * g + e]) - D) * kScale;
        }
        const uint32_t off = (c >> 1) * kTile + sw_off(i, (c & 1) * 4 + g);
        st_shared4(p_base + off, pack_bf16x2(pv[0], pv[1]), pack_bf16x2(pv[2], pv[3]), pack_bf16x2(pv[4], pv[5]),
                   pack_bf16x2(pv[6], pv[7]));
        st_shared4(ds_base + off, pack_bf16x2(dv[0], dv[1]), pack_bf16x2(dv[2], dv[3]), pack_bf16x2(dv[4], dv[5]),
                   pack_bf16x2(dv[6], dv[7]));
      }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // P, dS visible to the tensor cores
    tc_fence_before();
    mbar_arrive(&bars[2]);
    if (!mbar_wait(&bars[3], 0)) atomicExch(p.err, 14);
    tc_fence_after();
    // TMEM row i holds dQ row i and dK / dV row j = i; each half of the
    // pair stores 32 of the 64 columns of each
    bf16* drow = p.out + size_t(row0 + i) * 3 * p.C;
#pragma unroll 1
    for (int t = 0; t < 3; ++t) {
      const uint32_t col = t == 0 ? 0u : (t == 1 ? 192u : 128u);     // dQ, dK, dV
      uint32_t r[32];
      tmem_ld32(trow + col + 32 * hf, r);
      if (live) store_row32(drow + t * p.C + h * 64 + 32 * hf, r, p.acc != 0);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256) : "memory");
  }
}

constexpr size_t kFwdSmem = 5 * kTile + 1024 + 64 + 4 * 128 * sizeof(float2);
constexpr size_t kBwdSmem = 7 * kTile + 1024;   // 115,712 B: two CTAs in an SM's 228 KB

}  // namespace

struct AttnTcPlan {
  AttnParams p;
};

bool attention_tc_ok(int L, int C, int heads) { return L >= 1 && L <= 128 && heads > 0 && C == 64 * heads; }

AttnTcPlan* attention_tc_plan(const void* qkv, const void* out, const void* dout, int B, int L, int C, int heads,
                              int* err) {
  if (!attention_tc_ok(L, C, heads)) return nullptr;
  AttnTcPlan* a = new AttnTcPlan();
  a->p = AttnParams{};
  a->p.L = L;
  a->p.C = C;
  a->p.heads = heads;
  a->p.err = err;
  a->p.o = static_cast<const bf16*>(out);
  const int64_t rows = int64_t(B) * L;
  if (!tc_encode_2d(&a->p.tm_qkv, qkv, rows, 3 * C, 128) ||
      (dout && !tc_encode_2d(&a->p.tm_do, dout, rows, C, 128))) {
    delete a;
    return nullptr;
  }
  // Both kernels are sized for two CTAs per SM, which needs the largest
  // shared-memory carveout (the default sizes the carveout for one block).
  if (cudaFuncSetAttribute(attn_fwd_tc_k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kFwdSmem)) !=
          cudaSuccess ||
      cudaFuncSetAttribute(attn_bwd_tc_k, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kBwdSmem)) !=
          cudaSuccess ||
      cudaFuncSetAttribute(attn_fwd_tc_k, cudaFuncAttributePreferredSharedMemoryCarveout,
                           int(cudaSharedmemCarveoutMaxShared)) != cudaSuccess ||
      cudaFuncSetAttribute(attn_bwd_tc_k, cudaFuncAttributePreferredSharedMemoryCarveout,
                           int(cudaSharedmemCarveoutMaxShared)) != cudaSuccess) {
    delete a;
    return nullptr;
  }
  return a;
}

void attention_tc_destroy(AttnTcPlan* a) { delete a; }

void attention_tc_fwd(const AttnTcPlan* a, const int32_t* len, void* out, float* lse, int B, cudaStream_t st) {
  AttnParams p = a->p;
  p.len = len;
  p.out = static_cast<bf16*>(out);
  p.lse = lse;
  p.acc = 0;
  launch_k(attn_fwd_tc_k, B * p.heads, kAttnThreads, kFwdSmem, st, p);
}

void attention_tc_bwd(const AttnTcPlan* a, const int32_t* len, const float* lse, void* dqkv, int B, bool acc,
                      cudaStream_t st) {
  AttnParams p = a->p;
  p.len = len;
  p.out = static_cast<bf16*>(dqkv);
  p.lse = const_cast<float*>(lse);
  p.acc = acc ? 1 : 0;
  launch_k(attn_bwd_tc_k, B * p.heads, kAttnThreads, kBwdSmem, st, p);
}

}  // namespace fo
