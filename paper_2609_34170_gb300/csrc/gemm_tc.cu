// Projection GEMM on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
//   out[m][n] (op)= sum_k X[m][k] * W[n][k]       X: activations [M][K] bf16
//                                                  W: weights     [N][K] bf16 (K-major)
//
// Swap-AB tiling: a tile is 128 weight rows (the MMA's M = 128 TMEM lanes) by
// BN tokens (the MMA's N, 32..256): with 50-66 tokens per robot the weights
// are the large operand, and one kernel covers both the bandwidth-bound
// batch-1 case (few tiles, split-K over the grid) and the compute-bound
// large-batch case (many 128 x 256 tiles).
//
// Warp roles (192 threads): warp 0 = TMA producer, warp 1 = TMEM allocator +
// single-thread MMA issuer, warps 2..5 = epilogue (warp w reads TMEM lanes
// 32*(w%4)..+31).  Operand tiles are 64 K-elements wide (one 128-byte
// swizzle row) in an S-stage shared-memory ring guarded by mbarriers.  Every
// wait is bounded: on timeout the kernel raises ERR_TIMEOUT in the device
// error word and unwinds instead of hanging.
//
// Work distribution:
//  * no split: CTAs walk the tiles (persistent when there are more tiles than
//    SMs) with two TMEM accumulators, so the epilogue of one tile overlaps the
//    MMAs of the next;
//  * few tiles: the K dimension is split over grid.z.  The splits of a tile
//    form a thread-block cluster; each writes its fp32 partial to L2, the
//    cluster barrier publishes them, and rank q sums a column slice over the
//    splits in order (deterministic) and applies the epilogue;
//  * workspace mode (no cluster, for callers that bring their own scratch):
//    the last split to arrive (per-tile counter) sums all partials.
// The epilogue stages each 16-token chunk in shared memory so that global
// stores are 16-byte row segments written by all 128 epilogue threads.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "launch.h"
#include "tc_common.cuh"

namespace ravel {
namespace {

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;
constexpr int TC_THREADS = 192;
constexpr uint32_t TC_A_BYTES = TC_BM * TC_BK * 2;
constexpr int TC_SMEM_BUDGET = 200 * 1024;   // operand ring
constexpr int TC_SMEM_MAX = 227 * 1024;
constexpr int STG_LD = 132;                  // staging pitch (floats): 16 tokens x 128 tile rows
constexpr uint32_t STG_BYTES = 16 * STG_LD * 4;

enum { RED_NONE = 0, RED_L2_CLUSTER = 1, RED_WORKSPACE = 2 };

struct TcParams {
  int M, N, K;
  int bn, stages, splits, num_kb;
  int reduce;           // how the splits of a tile are combined (splits > 1)
  uint32_t ring_bytes;  // operand ring bytes (1024-aligned)
  uint32_t acc_cols;    // TMEM columns of one accumulator
  int tiles_n, tiles_m, num_tiles;
  int epi;              // Epi
  int out_bf16;
  void* out;
  int ldo;
  const float* bias;
  float* ws;
  int* counters;
  int* err;
  bf16* vt;
  int v_col0, vt_hd, vt_tokens, vt_kvp, vt_hkv;
};

// The i-th work item of this CTA: a tile (tn, tm) and split sp.  With splits
// the grid is (tiles_n, tiles_m, splits) and every CTA has one item; without,
// the grid is 1-D and CTA c takes tiles c, c + gridDim.x, ... (token tiles of
// one weight tile are adjacent, so concurrently running CTAs share it in L2).
__device__ __forceinline__ bool work_item(const TcParams& p, int i, int& tn, int& tm, int& sp) {
  if (p.splits > 1) {
    if (i) return false;
    tn = blockIdx.x;
    tm = blockIdx.y;
    sp = blockIdx.z;
    return true;
  }
  const int t = blockIdx.x + i * gridDim.x;
  if (t >= p.num_tiles) return false;
  tm = t % p.tiles_m;
  tn = t / p.tiles_m;
  sp = 0;
  return true;
}

// dst[k] = bf16(vals[k] + add) for k < n (n <= 16), with 2-, 4-, 8- or
// 16-byte stores as alignment allows.
__device__ __forceinline__ void store_bf16_run(bf16* dst, const float* vals, int n, float add) {
  int k = 0;
  while (k < n) {
    const uintptr_t a = (uintptr_t)(dst + k);
    if ((a & 15) == 0 && n - k >= 8) {
      *(uint4*)(dst + k) = make_uint4(pack_bf16x2(vals[k] + add, vals[k + 1] + add),
                                      pack_bf16x2(vals[k + 2] + add, vals[k + 3] + add),
                                      pack_bf16x2(vals[k + 4] + add, vals[k + 5] + add),
                                      pack_bf16x2(vals[k + 6] + add, vals[k + 7] + add));
      k += 8;
    } else if ((a & 7) == 0 && n - k >= 4) {
      *(uint2*)(dst + k) = make_uint2(pack_bf16x2(vals[k] + add, vals[k + 1] + add),
                                      pack_bf16x2(vals[k + 2] + add, vals[k + 3] + add));
      k += 4;
    } else if ((a & 3) == 0 && n - k >= 2) {
      *(uint32_t*)(dst + k) = pack_bf16x2(vals[k] + add, vals[k + 1] + add);
      k += 2;
    } else {
      dst[k] = __float2bfloat16_rn(vals[k] + add);
      k += 1;
    }
  }
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// v[4g + e] += sum over splits s = 0..S-1 (in order) of the partial of this
// thread's row at column group g (g < NG); b0 points at split 0, group 0;
// splits are sstride floats apart, groups 512.  Up to 16 float4 loads are in
// flight per batch; splits past S add exact zeros.
template <int NG>
__device__ __forceinline__ void reduce_splits_l2(const float* b0, int S, size_t sstride, float v[16]) {
  constexpr int GB = 16 / NG;
  for (int s0 = 0; s0 < S; s0 += GB) {
    float4 x[GB][NG];
#pragma unroll
    for (int u = 0; u < GB; ++u)
#pragma unroll
      for (int g = 0; g < NG; ++g)
        x[u][g] = (s0 + u < S) ? __ldcg((const float4*)(b0 + (size_t)(s0 + u) * sstride + (size_t)g * 512))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int u = 0; u < GB; ++u)
#pragma unroll
      for (int g = 0; g < NG; ++g) {
        v[4 * g] += x[u][g].x;
        v[4 * g + 1] += x[u][g].y;
        v[4 * g + 2] += x[u][g].z;
        v[4 * g + 3] += x[u][g].w;
      }
  }
}

// Epilogue of tokens m0 .. m0+nc-1 (nc <= 16) of tile row block tile_n: v[i]
// is this thread's tile row r at token m0+i.  All 128 epilogue threads call it
// together.  The chunk is transposed through `stage` so that each thread then
// writes one token's 16 (or, for GeGLU, 8) consecutive outputs as 16-byte
// stores.  The V columns of the QKV projection also go out transposed.
__device__ __forceinline__ void epilogue_chunk(const TcParams& p, int tile_n, int m0, int nc, int r,
                                               const float v[16], float* stage) {
#pragma unroll
  for (int i = 0; i < 16; ++i) stage[i * STG_LD + r] = v[i];
  if (p.vt) {
    // this thread's feature is one row d of V^T: its tokens m0.. are
    // consecutive keys of at most two robots -> vectorised runs
    const int n = tile_n * TC_BM + r;
    if (n >= p.v_col0 && n < p.N) {
      const float bb = p.bias ? p.bias[n] : 0.f;
      const int g = (n - p.v_col0) / p.vt_hd, d = (n - p.v_col0) % p.vt_hd;
      const int nv = min(nc, p.M - m0);
      int i = 0;
      while (i < nv) {
        const int m = m0 + i;
        const int rb = m / p.vt_tokens, kk = m % p.vt_tokens;
        const int run = min(nv - i, p.vt_tokens - kk);
        bf16* dst = p.vt + ((size_t)(rb * p.vt_hkv + g) * p.vt_hd + d) * p.vt_kvp + kk;
        store_bf16_run(dst, v + i, run, bb);
        i += run;
      }
    }
  }
  epi_bar();
  const int c = r >> 3, fg = r & 7;
  const int m = m0 + c;
  if (c < nc && m < p.M) {
    const float* srow = stage + c * STG_LD;
    if (p.epi == EPI_GEGLU) {
      // rows 0..63 of the tile are gate features, rows 64..127 the matching up features
      const int f0 = tile_n * 64 + fg * 8, nf = p.N / 2;
      float o[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) o[q] = gelu_tanh_f(srow[fg * 8 + q]) * srow[64 + fg * 8 + q];
      bf16* dst = (bf16*)p.out + (size_t)m * p.ldo + f0;
      if (f0 + 8 <= nf && ((uintptr_t)dst & 15) == 0) {
        *(uint4*)dst = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]), pack_bf16x2(o[4], o[5]),
                                  pack_bf16x2(o[6], o[7]));
      } else {
        for (int q = 0; q < 8; ++q)
          if (f0 + q < nf) dst[q] = __float2bfloat16_rn(o[q]);
      }
    } else {
      const int n0 = tile_n * TC_BM + fg * 16;
      const bool full = n0 + 16 <= p.N;
      float x[16];
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        x[q] = srow[fg * 16 + q] + ((p.bias && n0 + q < p.N) ? p.bias[n0 + q] : 0.f);
        if (p.epi == EPI_STORE_SILU) x[q] = silu_f(x[q]);
      }
      if (p.epi == EPI_ADD_F32) {
        float* dst = (float*)p.out + (size_t)m * p.ldo + n0;
        if (full && ((uintptr_t)dst & 15) == 0) {
          float4 a[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) a[k] = *(const float4*)(dst + 4 * k);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            *(float4*)(dst + 4 * k) =
                make_float4(a[k].x + x[4 * k], a[k].y + x[4 * k + 1], a[k].z + x[4 * k + 2], a[k].w + x[4 * k + 3]);
        } else {
          for (int q = 0; q < 16; ++q)
            if (n0 + q < p.N) dst[q] += x[q];
        }
      } else if (p.out_bf16) {
        bf16* dst = (bf16*)p.out + (size_t)m * p.ldo + n0;
        if (full && ((uintptr_t)dst & 15) == 0) {
          *(uint4*)dst = make_uint4(pack_bf16x2(x[0], x[1]), pack_bf16x2(x[2], x[3]), pack_bf16x2(x[4], x[5]),
                                    pack_bf16x2(x[6], x[7]));
          *(uint4*)(dst + 8) = make_uint4(pack_bf16x2(x[8], x[9]), pack_bf16x2(x[10], x[11]),
                                          pack_bf16x2(x[12], x[13]), pack_bf16x2(x[14], x[15]));
        } else {
          for (int q = 0; q < 16; ++q)
            if (n0 + q < p.N) dst[q] = __float2bfloat16_rn(x[q]);
        }
      } else {
        float* dst = (float*)p.out + (size_t)m * p.ldo + n0;
        if (full && ((uintptr_t)dst & 15) == 0) {
#pragma unroll
          for (int k = 0; k < 4; ++k)
            *(float4*)(dst + 4 * k) = make_float4(x[4 * k], x[4 * k + 1], x[4 * k + 2], x[4 * k + 3]);
        } else {
          for (int q = 0; q < 16; ++q)
            if (n0 + q < p.N) dst[q] = x[q];
        }
      }
    }
  }
  epi_bar();
}

__global__ void __launch_bounds__(TC_THREADS, 2)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX, TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int BN = p.bn, S = p.stages;
  const uint32_t b_bytes = (uint32_t)BN * TC_BK * 2;
  uint8_t* a_s = smem;
  uint8_t* b_s = smem + (size_t)S * TC_A_BYTES;
  uint64_t* full = (uint64_t*)(smem + p.ring_bytes);
  uint64_t* empty = full + S;
  uint64_t* acc_full = empty + S;      // [2]
  uint64_t* acc_empty = acc_full + 2;  // [2]
  uint32_t* tmem_slot = (uint32_t*)(acc_empty + 2);
  int* flags = (int*)(tmem_slot + 1);   // [0] abort, [1] last split, [2] issued, [3] consumed
  float* stage = (float*)(((uintptr_t)(flags + 4) + 15) & ~(uintptr_t)15);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t ncols = (p.splits > 1) ? p.acc_cols : 2 * p.acc_cols;
  int tn0 = 0, tm0 = 0, sp0 = 0;
  const bool has_work = work_item(p, 0, tn0, tm0, sp0);
  const int kb0_first = (int)((long)sp0 * p.num_kb / p.splits);
  const int kb1_first = (int)((long)(sp0 + 1) * p.num_kb / p.splits);
  const int npre = has_work ? min(S, kb1_first - kb0_first) : 0;

  pdl_trigger();
  uint64_t pol_w = 0, pol_x = 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 128);
    }
    flags[0] = flags[1] = flags[2] = flags[3] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    // Weights never depend on earlier kernels: stream the first stages' weight
    // tiles while the previous kernel is still finishing.
    asm volatile("prefetch.tensormap [%0];" ::"l"(&tmW) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(&tmX) : "memory");
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol_w));
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol_x));
    for (int i = 0; i < npre; ++i) {
      mbar_expect_tx(&full[i], TC_A_BYTES + b_bytes);
      tma_load_2d(&tmW, &full[i], a_s + (size_t)i * TC_A_BYTES, (kb0_first + i) * TC_BK, tn0 * TC_BM, pol_w);
    }
  }
  // everything below may read what earlier kernels wrote; TMEM is taken only
  // now, so a CTA waiting here never holds columns its predecessor needs
  pdl_wait();
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  cta_sync();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      int it = 0;   // ring position across all work items
      bool ok = true;
      int tn, tm, sp;
      for (int i = 0; ok && work_item(p, i, tn, tm, sp); ++i) {
        const int kb0 = (int)((long)sp * p.num_kb / p.splits), kb1 = (int)((long)(sp + 1) * p.num_kb / p.splits);
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int s = it % S;
          if (it < npre) {   // weight tile already in flight
            tma_load_2d(&tmX, &full[s], b_s + (size_t)s * b_bytes, kb * TC_BK, tm * BN, pol_x);
            continue;
          }
          if (!mbar_wait(&empty[s], ((uint32_t)(it / S) & 1u) ^ 1u)) {
            flags[0] = 1;
            ok = false;
            break;
          }
          mbar_expect_tx(&full[s], TC_A_BYTES + b_bytes);
          tma_load_2d(&tmW, &full[s], a_s + (size_t)s * TC_A_BYTES, kb * TC_BK, tn * TC_BM, pol_w);
          tma_load_2d(&tmX, &full[s], b_s + (size_t)s * b_bytes, kb * TC_BK, tm * BN, pol_x);
        }
      }
      flags[2] = it;
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(TC_BM, BN);
      int it = 0;
      bool ok = true;
      int tn, tm, sp;
      for (int i = 0; ok && work_item(p, i, tn, tm, sp); ++i) {
        const int b = i & 1;
        // the accumulator of item i - 2 must have been drained by the epilogue
        if (i >= 2 && !mbar_wait(&acc_empty[b], (uint32_t)((i >> 1) - 1) & 1u)) {
          flags[0] = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)b * p.acc_cols;
        const int kb0 = (int)((long)sp * p.num_kb / p.splits), kb1 = (int)((long)(sp + 1) * p.num_kb / p.splits);
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int s = it % S;
          if (!mbar_wait(&full[s], (uint32_t)(it / S) & 1u)) {
            flags[0] = 1;
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = sw128_desc(smem_u32(a_s + (size_t)s * TC_A_BYTES));
          const uint64_t bd = sw128_desc(smem_u32(b_s + (size_t)s * b_bytes));
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k)
            umma_bf16(d, ad + 2 * k, bd + 2 * k, idesc, (kb > kb0 || k > 0) ? 1u : 0u);
          umma_commit(&empty[s]);
        }
        umma_commit(&acc_full[b]);   // arrives once every MMA issued above has completed
      }
      flags[3] = it;
    }
    __syncwarp();
  } else {
    // epilogue warps 2..5: TMEM lane quarter q = warp % 4, tile row r
    const int q = warp & 3;
    const int r = q * 32 + lane;
    int tn, tm, sp;
    for (int i = 0; work_item(p, i, tn, tm, sp); ++i) {
      const int b = i & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[b], (uint32_t)(i >> 1) & 1u));
      if (!ok) {
        if (lane == 0) flags[0] = 1;
        break;
      }
      tc_fence_after();
      const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)b * p.acc_cols;
      const int m_base = tm * BN;
      if (p.splits == 1) {
        for (int c0 = 0; c0 < BN; c0 += 16) {
          float v[16];
          tmem_ld16(trow + c0, v);
          if (c0 + 16 >= BN) {   // accumulator drained: the MMA warp may reuse it
            tc_fence_before();
            mbar_arrive(&acc_empty[b]);
          }
          epilogue_chunk(p, tn, m_base + c0, 16, r, v, stage);
        }
      } else if (p.reduce == RED_L2_CLUSTER) {
        // this split's fp32 partial to the workspace as [col/4][row][4]: each
        // thread stores float4 of 4 consecutive columns, a warp one 512-byte run
        const size_t cl = (size_t)tm * gridDim.x + tn;
        float* w = p.ws + ((cl * p.splits + sp) * (size_t)(BN / 4)) * (TC_BM * 4) + (size_t)r * 4;
        for (int c0 = 0; c0 < BN; c0 += 16) {
          float v[16];
          tmem_ld16(trow + c0, v);
#pragma unroll
          for (int qq = 0; qq < 4; ++qq)
            __stcg((float4*)(w + (size_t)(c0 / 4 + qq) * (TC_BM * 4)),
                   make_float4(v[4 * qq], v[4 * qq + 1], v[4 * qq + 2], v[4 * qq + 3]));
        }
        __threadfence();
      } else {
        // workspace mode: [split][tile][col][row] partials, last arrival reduces
        const int tiles = gridDim.x * gridDim.y;
        const int tile_id = tm * gridDim.x + tn;
        for (int c0 = 0; c0 < BN; c0 += 16) {
          float v[16];
          tmem_ld16(trow + c0, v);
          float* w = p.ws + ((size_t)(sp * tiles + tile_id) * BN + c0) * TC_BM + r;
#pragma unroll
          for (int k = 0; k < 16; ++k) __stcg(w + (size_t)k * TC_BM, v[k]);
        }
        __threadfence();
        epi_bar();
        if (threadIdx.x == 64) {
          const int prev = atomicAdd(&p.counters[tile_id], 1);
          flags[1] = (prev == p.splits - 1);
        }
        epi_bar();
        if (flags[1]) {
          __threadfence();
          for (int c0 = 0; c0 < BN; c0 += 16) {
            float v[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) v[k] = 0.f;
            for (int s = 0; s < p.splits; ++s) {
              const float* w = p.ws + ((size_t)(s * tiles + tile_id) * BN + c0) * TC_BM + r;
              float x[16];
#pragma unroll
              for (int k = 0; k < 16; ++k) x[k] = __ldcg(w + (size_t)k * TC_BM);
#pragma unroll
              for (int k = 0; k < 16; ++k) v[k] += x[k];
            }
            epilogue_chunk(p, tn, m_base + c0, 16, r, v, stage);
          }
          if (threadIdx.x == 64) p.counters[tile_id] = 0;
        }
      }
    }
  }
  tc_fence_before();
  cta_sync();
  if (flags[0]) {
    // unwind: wait (bounded) for the copies this CTA issued but never consumed
    if (threadIdx.x == 0) {
      for (int i = flags[3]; i < flags[2]; ++i) mbar_wait(&full[i % S], (uint32_t)(i / S) & 1u);
      raise_error(p.err, ERR_TIMEOUT);
    }
    cta_sync();
  }
  if (p.reduce == RED_L2_CLUSTER && p.splits > 1) {
    // Every split of this tile has written its partial; the cluster barrier
    // (release / acquire) makes them visible.  Rank q sums columns
    // [q*BN/S, (q+1)*BN/S) over the splits in order and applies the epilogue.
    cluster_sync();
    if (warp >= 2) {
      const int r = (warp & 3) * 32 + lane;
      const int Sp = p.splits;
      const int cpr = BN / Sp;   // a multiple of 4
      const int rank = (int)cluster_ctarank();
      const size_t cl = (size_t)tm0 * gridDim.x + tn0;
      const float* base = p.ws + (cl * Sp * (size_t)(BN / 4) + rank * cpr / 4) * (TC_BM * 4) + (size_t)r * 4;
      const size_t sstride = (size_t)(BN / 4) * (TC_BM * 4);
      for (int cc = 0; cc < cpr; cc += 16) {
        const int nc = min(16, cpr - cc);
        float v[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = 0.f;
        const float* b0 = base + (size_t)(cc / 4) * (TC_BM * 4);
        if (nc == 16) reduce_splits_l2<4>(b0, Sp, sstride, v);
        else if (nc == 12) reduce_splits_l2<3>(b0, Sp, sstride, v);
        else if (nc == 8) reduce_splits_l2<2>(b0, Sp, sstride, v);
        else reduce_splits_l2<1>(b0, Sp, sstride, v);
        epilogue_chunk(p, tn0, tm0 * BN + rank * cpr + cc, nc, r, v, stage);
      }
    }
  }
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols) : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

cudaError_t get_encoder() {
  if (g_encode) return cudaSuccess;
  cudaDriverEntryPointQueryResult q;
  void* fn = nullptr;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
  if (e != cudaSuccess) return e;
  if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorSymbolNotFound;
  g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  return cudaSuccess;
}

// 2D bf16 map over a row-major [rows][cols] matrix (row stride ld elements),
// box = box_rows x 64 columns, 128-byte swizzle, zero fill out of bounds.
cudaError_t encode_2d(CUtensorMap* m, const void* base, int rows, int cols, int ld, int box_rows) {
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  cuuint32_t box[2] = {(cuuint32_t)TC_BK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Token-tile width: the smallest of 32/64/96/128 that holds M; beyond 128
// tokens, the multiple of 16 in [128, 256] whose tile count fills whole waves
// of the SMs best (per-CTA work ~ waves x BN), larger BN on ties.
int pick_bn(int M, int tiles_n, int num_sms) {
  const int cands[] = {32, 64, 96, 128};
  for (int c : cands)
    if (M <= c) return c;
  int best = 256;
  long best_cost = -1;
  for (int bn = 256; bn >= 128; bn -= 16) {
    const long tiles = (long)tiles_n * ((M + bn - 1) / bn);
    const long waves = (tiles + num_sms - 1) / num_sms;
    const long cost = waves * bn;
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

int g_max_cluster = 8;   // largest power-of-two cluster the split-K reduction may use

}  // namespace

cudaError_t init_tc_gemm() {
  cudaError_t e = get_encoder();
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(tc_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, TC_SMEM_MAX);
  if (e != cudaSuccess) return e;
  // clusters of 16 are beyond the portable limit: use them only if allowed
  if (cudaFuncSetAttribute(tc_gemm_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 1;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 16;
    cfg.gridDim = dim3(1, 1, 16);
    cfg.blockDim = dim3(TC_THREADS);
    cfg.dynamicSmemBytes = TC_SMEM_MAX;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, tc_gemm_kernel, &cfg) == cudaSuccess && n > 0) g_max_cluster = 16;
  }
  cudaGetLastError();
  return cudaSuccess;
}

bool tc_gemm_supported(const GemmArgs& g) {
  // TMA: 16-byte aligned bases and row strides
  if (g.K % 8 || g.lda % 8 || g.ldw % 8) return false;
  if (((uintptr_t)g.A & 15) || ((uintptr_t)g.W & 15)) return false;
  if (g.epi == EPI_GEGLU && (g.N % 128)) return false;
  return g.M > 0 && g.N > 0 && g.K > 0;
}

cudaError_t launch_gemm_tc(const GemmArgs& g, const TcWorkspace& ws, int num_sms, cudaStream_t st, bool cluster) {
  if (!g_encode) return cudaErrorInitializationError;
  const int tiles_n = (g.N + TC_BM - 1) / TC_BM;
  const int bn = pick_bn(g.M, tiles_n, num_sms);
  const int tiles_m = (g.M + bn - 1) / bn;
  const int num_kb = (g.K + TC_BK - 1) / TC_BK;
  const int tiles = tiles_n * tiles_m;
  int splits = 1;
  if (tiles < num_sms) splits = std::min(num_kb, std::max(1, num_sms / tiles));
  if (cluster) {
    // the splits of a tile form one cluster: a power of two, at most the cluster
    // limit, whose partials fit the workspace and whose column slices are
    // multiples of 4
    int c = 1;
    while (c * 2 <= std::min(splits, g_max_cluster) && (bn / (c * 2)) % 4 == 0 &&
           (size_t)(c * 2) * tiles * bn * TC_BM * 4 <= ws.ws_bytes)
      c *= 2;
    splits = c;
  } else {
    while (splits > 1 && ((size_t)splits * tiles * bn * TC_BM * 4 > ws.ws_bytes || tiles > ws.n_counters)) --splits;
  }
  const int reduce = splits == 1 ? RED_NONE : (cluster ? RED_L2_CLUSTER : RED_WORKSPACE);
  uint32_t acc_cols = 32;
  while ((int)acc_cols < bn) acc_cols <<= 1;
  const int stage_bytes = TC_A_BYTES + bn * TC_BK * 2;
  const int kb_per_item = (num_kb + splits - 1) / splits;
  const int grid_ctas = splits > 1 ? tiles * splits : std::min(tiles, num_sms);
  const int items = splits > 1 ? 1 : (tiles + grid_ctas - 1) / grid_ctas;
  int stages = std::min(8, TC_SMEM_BUDGET / stage_bytes);
  stages = std::max(2, std::min(stages, std::max(2, kb_per_item * items)));
  const size_t ring = ((size_t)stages * stage_bytes + 1023) / 1024 * 1024;
  // alignment slack + ring + barriers / TMEM slot / flags + staging tile (+ slack)
  const size_t smem = 1024 + ring + (2 * stages + 4) * 8 + 32 + 16 + STG_BYTES + 64;
  CUtensorMap mw, mx;
  cudaError_t e = encode_2d(&mw, g.W, g.N, g.K, g.ldw, TC_BM);
  if (e == cudaSuccess) e = encode_2d(&mx, g.A, g.M, g.K, g.lda, bn);
  if (e != cudaSuccess) return e;
  TcParams p{g.M, g.N, g.K, bn, stages, splits, num_kb, reduce, (uint32_t)ring, acc_cols, tiles_n, tiles_m, tiles,
             (int)g.epi, g.out_dt == DT_BF16 ? 1 : 0, g.out, g.ldo, g.bias, ws.ws, ws.counters, ws.err, (bf16*)g.vt,
             g.v_col0, g.vt_hd, g.vt_tokens, g.vt_kvp, g.vt_hkv};
  const dim3 grid = splits > 1 ? dim3(tiles_n, tiles_m, splits) : dim3(grid_ctas);
  return launch_kernel(tc_gemm_kernel, grid, dim3(TC_THREADS), smem, st,
                       reduce == RED_L2_CLUSTER ? (unsigned)splits : 1u, mw, mx, p);
}

}  // namespace ravel
