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
//    MMAs of the next; where the tiles are many, pairs of CTAs run 256-row
//    tiles with the two-SM MMA instead (tc_gemm_pair_kernel, below);
//  * few tiles: the K dimension is split over grid.z.  The splits of a tile
//    form a thread-block cluster and rank q sums a token slice over the splits
//    in order (deterministic) and applies the epilogue.  The partials travel
//    by st.async straight into rank q's shared memory, completing on an
//    mbarrier there (slices of up to 32 tokens), else through L2 and the
//    cluster barrier;
//  * workspace mode (no cluster, for callers that bring their own scratch):
//    the last split to arrive (per-tile counter) sums all partials.
// Epilogue: a chunk of tokens is written into a shared-memory box in the
// output layout and leaves through one TMA store (or a TMA reduce-add for the
// residual-stream epilogue), double-buffered so that the epilogue threads
// never wait on global memory; the workspace mode (and unaligned outputs)
// store from the threads instead.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <cstring>
#include <vector>

#include "common.cuh"
#include "kernels.h"
#include "launch.h"
#include "tc_common.cuh"

namespace ravel {
namespace {

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;
constexpr int TC_THREADS = 192;
constexpr int TC_PAIR_THREADS = 320;   // pair kernel: TMA, MMA and two sets of four epilogue warps
constexpr uint32_t TC_A_BYTES = TC_BM * TC_BK * 2;
constexpr int TC_SMEM_BUDGET = 200 * 1024;   // operand ring
constexpr int TC_SMEM_MAX = 227 * 1024;
constexpr int TC_RING_SPLIT = 128 * 1024;    // operand ring of a split-K launch
constexpr int STG_LD = 132;                  // SIMT staging pitch (floats): 16 tokens x 128 tile rows
constexpr uint32_t STG_BYTES = 16 * STG_LD * 4;
constexpr uint32_t XCH_BYTES = 32 * STG_LD * 4;  // GeGLU transpose tile (TMA epilogue): <= 32 tokens x 128 rows

enum { RED_NONE = 0, RED_L2_CLUSTER = 1, RED_WORKSPACE = 2, RED_DSMEM = 3, RED_DSMEM32 = 4 };
// Epilogue kind of an instantiation: outputs through TMA boxes as fp32, bf16,
// a reduce-add into the fp32 residual stream or the GeGLU pair -- fixed, so
// that a long persistent launch carries only the code of its own epilogue --
// or any of these chosen at run time (EK_TMA_ANY: the
// short split-K launches of one step then all run one binary, whose code the
// previous launch has left in the SM's instruction cache), or stored by the
// threads (EK_GENERIC: any epilogue; unaligned outputs and the workspace
// reduction).
enum { EK_F32 = 0, EK_BF16 = 1, EK_ADD = 2, EK_GEGLU = 3, EK_GENERIC = 4, EK_TMA_ANY = 5 };


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
  int tma_out;          // outputs leave through TMA boxes
  int oneshot;          // split launch whose whole K range fits the ring: tmW / tmX are 3-D maps
                        // (64, rows, K / 64) and one box each brings all of its k-tiles
  int box_m;            // tokens per epilogue chunk (= rows of a TMA output box)
  uint32_t box_bytes;   // bytes of one TMA output box (1024-aligned)
  uint32_t stg_off;     // SIMT transpose tile, or two TMA output boxes
  uint32_t xch_off;     // GeGLU exchange
  uint32_t rcv_off;     // RED_DSMEM*: the partials received from the splits, [split][cpr / 4][128 rows]
                        // float4, overlaid on the operand ring (free once every CTA of the cluster
                        // has finished its MMAs), else on the output boxes + exchange (used only
                        // after the sum)
  uint32_t bar_off;     // mbarriers, TMEM slot, flags
  unsigned long long wait_ns;   // limit of every bounded wait (ERR_TIMEOUT after it)
  int withhold;         // fault injection (tests): the MMA thread first waits for an arrival that
                        // nobody makes, so the launch gives up after wait_ns and unwinds
  const int* skip;      // optional device flag read after the dependency wait: nonzero -> the launch
                        // completes the copies it started and exits without computing
  uint32_t set_bytes;   // pair kernel: bytes from epilogue set 0's boxes / exchange to set 1's
};

// The TMA epilogue kind of a launch (EK_F32 .. EK_GEGLU).
__device__ __forceinline__ int tma_kind(const TcParams& p) {
  return p.epi == EPI_GEGLU ? EK_GEGLU : p.epi == EPI_ADD_F32 ? EK_ADD : p.out_bf16 ? EK_BF16 : EK_F32;
}

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

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }
// the 128 threads of epilogue warp set `set` (the pair kernel runs two sets)
__device__ __forceinline__ void epi_bar_set(int set) {
  if (set) asm volatile("bar.sync 2, 128;" ::: "memory");
  else asm volatile("bar.sync 1, 128;" ::: "memory");
}

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

// v[4g + e] (g < NG <= 8: up to 32 tokens) = sum over splits s = 0..S-1 (in
// order) of this thread's row at column group g; as reduce_splits_l2, with up
// to 24 float4 loads in flight per batch (one batch for every launch here).
template <int NG>
__device__ __forceinline__ void reduce_slice_l2(const float* b0, int S, size_t sstride, float v[32]) {
  constexpr int GB = (24 / NG) > 0 ? 24 / NG : 1;
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

// v[4g + e] (g < NG <= 8) = sum over splits s = 0..S-1 (in order) of the
// received bf16 partials: b0 points at this thread's four tokens of split 0,
// group 0 (half of a two-row message); group g of split s is (s * NG + g) *
// 128 uint2 further.
template <int NG>
__device__ __forceinline__ void reduce_slice_smem(const uint2* b0, int S, float v[32]) {
  #pragma unroll 1
  for (int s = 0; s < S; ++s) {
    uint2 x[NG];
#pragma unroll
    for (int g = 0; g < NG; ++g) x[g] = b0[(size_t)(s * NG + g) * TC_BM];
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      v[4 * g] += __uint_as_float(x[g].x << 16);
      v[4 * g + 1] += __uint_as_float(x[g].x & 0xFFFF0000u);
      v[4 * g + 2] += __uint_as_float(x[g].y << 16);
      v[4 * g + 3] += __uint_as_float(x[g].y & 0xFFFF0000u);
    }
  }
}

// As above for fp32 partials: b0 points at this thread's row of split 0,
// group 0; group g of split s is (s * NG + g) * 128 float4 further.
template <int NG>
__device__ __forceinline__ void reduce_slice_smem(const float4* b0, int S, float v[32]) {
  #pragma unroll 1
  for (int s = 0; s < S; ++s) {
    float4 x[NG];
#pragma unroll
    for (int g = 0; g < NG; ++g) x[g] = b0[(size_t)(s * NG + g) * TC_BM];
#pragma unroll
    for (int g = 0; g < NG; ++g) {
      v[4 * g] += x[g].x;
      v[4 * g + 1] += x[g].y;
      v[4 * g + 2] += x[g].z;
      v[4 * g + 3] += x[g].w;
    }
  }
}

// Epilogue of tokens m0 .. m0+nc-1 (nc <= 16) of tile row block tile_n: v[i]
// is this thread's tile row r at token m0+i.  All 128 epilogue threads call it
// together.  The chunk is transposed through `stage` so that each thread then
// writes one token's 16 (or, for GeGLU, 8) consecutive outputs as 16-byte
// stores.
__device__ __forceinline__ void epilogue_chunk(const TcParams& p, int tile_n, int m0, int nc, int r,
                                               const float v[16], float* stage) {
#pragma unroll
  for (int i = 0; i < 16; ++i) stage[i * STG_LD + r] = v[i];
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
      for (int q = 0; q < 8; ++q) {
        const int ng = tile_n * TC_BM + fg * 8 + q;   // gate row; its up row is ng + 64
        const float bg = p.bias ? p.bias[ng] : 0.f, bu = p.bias ? p.bias[ng + 64] : 0.f;
        o[q] = gelu_tanh_bf16out(srow[fg * 8 + q] + bg) * (srow[64 + fg * 8 + q] + bu);
      }
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


// TMA epilogue of tokens m0 .. m0+box_m-1 of tile row block tile_n: v[i] is
// this thread's tile row r at token m0+i, brow its bias.  All 128 epilogue
// threads call it together.  The chunk is written into output box `ebuf` in
// shared memory (token-major, as the output), and thread 64 sends the box
// with one TMA store (EPI_ADD_F32: TMA reduce-add into the residual stream);
// rows past M and columns past N are clipped by the tensor map.
// f(i) for i < n (n <= NV, a multiple of G), unrolled: without a bound
// check when n == NV, else one per group of G (the epilogue warps run one per
// scheduler, so every compare and branch in these loops is exposed latency)
template <int NV, int G = 4, typename F>
__device__ __forceinline__ void for_upto(int n, F&& f) {
  static_assert(NV % G == 0, "whole groups");
  if (n == NV) {
#pragma unroll
    for (int i = 0; i < NV; ++i) f(i);
  } else {
#pragma unroll
    for (int g = 0; g < NV; g += G) {
      if (g >= n) break;
#pragma unroll
      for (int i = g; i < g + G; ++i) f(i);
    }
  }
}

template <int EK, int NV = 16>
__device__ __forceinline__ void epilogue_tma(const TcParams& p, const CUtensorMap* tmO, int tile_n, int m0, int r,
                                             const float* v, float brow, uint8_t* boxes, float* xch, int& ebuf) {
  const int bm = p.box_m;   // <= NV
  // epilogue warp set (threads 64..191: 0; 192..319: 1, pair kernel only) and
  // the thread of the set that issues and waits for its TMA stores
  const int set = threadIdx.x >= 192 ? 1 : 0;
  const bool issuer = threadIdx.x == 64 + 128 * set;
  // the box written two chunks ago must have been read by its TMA store
  if (issuer) bulk_wait_read<1>();
  epi_bar_set(set);
  uint8_t* box = boxes + (size_t)ebuf * p.box_bytes;
  const int kind = EK == EK_TMA_ANY ? tma_kind(p) : EK;   // a constant in the fixed-kind instantiations
  if (kind == EK_GEGLU) {
    // tile rows 0..63 are gate features, 64..127 the matching up features:
    // transpose through xch so that every thread then forms 8 outputs of one
    // token (the GELUs spread over all 128 threads)
    for_upto<NV>(bm, [&](int i) { xch[i * STG_LD + r] = v[i] + brow; });
    epi_bar_set(set);
#pragma unroll
    for (int h = 0; h < NV / 16; ++h) {
      const int c = (r >> 3) + 16 * h, fg = r & 7;
      if (c < bm) {
        const float4* g4 = (const float4*)(xch + c * STG_LD + fg * 8);
        const float4* u4 = (const float4*)(xch + c * STG_LD + 64 + fg * 8);
        const float4 ga = g4[0], gb = g4[1], ua = u4[0], ub = u4[1];
        *(uint4*)((bf16*)box + c * 64 + fg * 8) =
            make_uint4(pack_bf16x2(gelu_tanh_bf16out(ga.x) * ua.x, gelu_tanh_bf16out(ga.y) * ua.y),
                       pack_bf16x2(gelu_tanh_bf16out(ga.z) * ua.z, gelu_tanh_bf16out(ga.w) * ua.w),
                       pack_bf16x2(gelu_tanh_bf16out(gb.x) * ub.x, gelu_tanh_bf16out(gb.y) * ub.y),
                       pack_bf16x2(gelu_tanh_bf16out(gb.z) * ub.z, gelu_tanh_bf16out(gb.w) * ub.w));
      }
    }
  } else if (kind == EK_BF16) {
    bf16* o = (bf16*)box;
    if (p.epi == EPI_STORE_SILU)
      for_upto<NV>(bm, [&](int i) { o[i * TC_BM + r] = __float2bfloat16_rn(silu_f(v[i] + brow)); });
    else
      for_upto<NV>(bm, [&](int i) { o[i * TC_BM + r] = __float2bfloat16_rn(v[i] + brow); });
  } else {
    float* o = (float*)box;
    if (kind == EK_F32 && p.epi == EPI_STORE_SILU)
      for_upto<NV>(bm, [&](int i) { o[i * TC_BM + r] = silu_f(v[i] + brow); });
    else
      for_upto<NV>(bm, [&](int i) { o[i * TC_BM + r] = v[i] + brow; });
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  epi_bar_set(set);
  if (issuer) {
    if (kind == EK_ADD) tma_reduce_add_2d(tmO, box, tile_n * TC_BM, m0);
    else tma_store_2d(tmO, box, kind == EK_GEGLU ? tile_n * 64 : tile_n * TC_BM, m0);
    bulk_commit();
  }
  ebuf ^= 1;
}

// RED = p.reduce and EK = the epilogue kind, fixed per instantiation so that
// each reduction mode gets its own register allocation and each launch only
// the code it runs.
template <int RED, int EK>
__global__ void __launch_bounds__(TC_THREADS, 2)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                   const __grid_constant__ CUtensorMap tmO, TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned; derived from smem_raw by pointer arithmetic so that the
  // compiler keeps it (and everything indexed from it) in the shared window
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int BN = p.bn, S = p.stages;
  const uint32_t b_bytes = (uint32_t)BN * TC_BK * 2;
  uint8_t* a_s = smem;
  uint8_t* b_s = smem + (size_t)S * TC_A_BYTES;
  uint8_t* stg_raw = smem + p.stg_off;
  float* stage = (float*)stg_raw;
  float* xch = (float*)(smem + p.xch_off);
  uint64_t* full = (uint64_t*)(smem + p.bar_off);
  uint64_t* empty = full + S;
  uint64_t* acc_full = empty + S;      // [2]
  uint64_t* acc_empty = acc_full + 2;  // [2]
  uint64_t* rcv_bar = acc_empty + 2;    // RED_DSMEM*: every split's slice of this rank has arrived
  uint32_t* tmem_slot = (uint32_t*)(rcv_bar + 1);
  int* flags = (int*)(tmem_slot + 1);   // [0] abort, [1] last split, [2] issued, [3] consumed

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t ncols = (p.splits > 1) ? p.acc_cols : 2 * p.acc_cols;
  int tn0 = 0, tm0 = 0, sp0 = 0;
  const bool has_work = work_item(p, 0, tn0, tm0, sp0);
  const int kb0_first = (int)((long)sp0 * p.num_kb / p.splits);
  const int kb1_first = (int)((long)(sp0 + 1) * p.num_kb / p.splits);
  const int npre = has_work ? min(S, kb1_first - kb0_first) : 0;
  const int cpr = BN / p.splits;   // tokens of the slice each split rank owns (a multiple of 4)
  constexpr bool TMA_OUT = EK != EK_GENERIC;
  // partials exchanged through distributed shared memory: RED_DSMEM in bf16
  // (two rows per message), RED_DSMEM32 in fp32
  constexpr bool DSM = RED == RED_DSMEM || RED == RED_DSMEM32;

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
    mbar_init(rcv_bar, 1);   // RED_DSMEM*: the partials' arrival; otherwise armed by nobody
    flags[0] = flags[1] = flags[2] = flags[3] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    // the slices of all splits (this one's included): 128 rows x cpr tokens each
    if constexpr (DSM) mbar_expect_tx(rcv_bar, (uint32_t)(BN * TC_BM * (RED == RED_DSMEM ? 2 : 4)));
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    // Weights never depend on earlier kernels: stream the first stages' weight
    // tiles while the previous kernel is still finishing.
    asm volatile("prefetch.tensormap [%0];" ::"l"(&tmW) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(&tmX) : "memory");
    if (TMA_OUT) asm volatile("prefetch.tensormap [%0];" ::"l"(&tmO) : "memory");
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol_w));
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol_x));
  }
  // A launch that may be skipped at run time (p.skip) issues nothing before
  // it has read its flag after the wait; every other launch streams its first
  // weight tiles now, while the previous kernel is still finishing.
  auto issue_weight_prologue = [&]() {
    if (p.oneshot) {
      // every weight k-tile of this CTA in one box; the token k-tiles follow
      // after the wait into the same barrier
      // (the boxes are S = the largest split's k-tile count deep; a shorter
      // split ignores the extra tile)
      mbar_expect_tx(&full[0], (uint32_t)S * (TC_A_BYTES + b_bytes));
      tma_load_3d(&tmW, &full[0], a_s, 0, tn0 * TC_BM, kb0_first, pol_w);
    } else {
      for (int i = 0; i < npre; ++i) {
        mbar_expect_tx(&full[i], TC_A_BYTES + b_bytes);
        tma_load_2d(&tmW, &full[i], a_s + (size_t)i * TC_A_BYTES, (kb0_first + i) * TC_BK, tn0 * TC_BM, pol_w);
      }
      // a split CTA has one short K range: the rest of its weight slice goes
      // to L2 now, so that after the wait every operand load is an L2 hit
      if (p.splits > 1)
        for (int kb = kb0_first + npre; kb < kb1_first; ++kb) prefetch_l2_2d(&tmW, kb * TC_BK, tn0 * TC_BM);
    }
  };
  if (threadIdx.x == 0 && !p.skip) issue_weight_prologue();
  // everything below may read what earlier kernels wrote; TMEM is taken only
  // now, so a CTA waiting here never holds columns its predecessor needs
  pdl_wait();
  if (p.skip) {
    // nothing is in flight yet; the flag is the same for every CTA
    if (*p.skip) return;
    if (threadIdx.x == 0) issue_weight_prologue();
  }
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
    if (lane == 0 && p.oneshot) {
      tma_load_3d(&tmX, &full[0], b_s, 0, tm0 * BN, kb0_first, pol_x);
      flags[2] = 1;
    } else if (lane == 0) {
      int it = 0;   // ring position across all work items
      bool ok = true;
      int tn, tm, sp;
      for (int i = 0; ok && work_item(p, i, tn, tm, sp); ++i) {
        const int kb0 = (int)((long)sp * p.num_kb / p.splits), kb1 = (int)((long)(sp + 1) * p.num_kb / p.splits);
        #pragma unroll 1
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int s = it % S;
          if (it < npre) {   // weight tile already in flight
            tma_load_2d(&tmX, &full[s], b_s + (size_t)s * b_bytes, kb * TC_BK, tm * BN, pol_x);
            continue;
          }
          if (!mbar_wait(&empty[s], ((uint32_t)(it / S) & 1u) ^ 1u, p.wait_ns)) {
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
    // RED_DSMEM*: one arrival per thread on the cluster barrier that opens the
    // exchange (the epilogue warps arrive once their MMAs are complete)
    if constexpr (DSM) cluster_arrive_release();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(TC_BM, BN);
      int it = 0;
      bool ok = true;
      int tn, tm, sp;
      // fault injection: an arrival that never comes (rcv_bar is armed by
      // nobody outside the RED_DSMEM modes, which the host never combines with this)
      if (p.withhold && !mbar_wait(rcv_bar, 0, p.wait_ns)) {
        flags[0] = 1;
        ok = false;
      }
      if (ok && p.oneshot) {   // one item, every k-tile behind one barrier
        ok = mbar_wait(&full[0], 0, p.wait_ns);
        if (ok) {
          tc_fence_after();
          #pragma unroll 1
          for (int kb = 0; kb < kb1_first - kb0_first; ++kb) {
            const uint64_t ad = sw128_desc(smem_u32(a_s + (size_t)kb * TC_A_BYTES));
            const uint64_t bd = sw128_desc(smem_u32(b_s + (size_t)kb * b_bytes));
#pragma unroll
            for (int k = 0; k < TC_BK / 16; ++k)
              umma_bf16(tmem, ad + 2 * k, bd + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          }
          umma_commit(&acc_full[0]);
          it = 1;
        } else {
          flags[0] = 1;
        }
      }
      for (int i = 0; !p.oneshot && ok && work_item(p, i, tn, tm, sp); ++i) {
        const int b = i & 1;
        // the accumulator of item i - 2 must have been drained by the epilogue
        if (i >= 2 && !mbar_wait(&acc_empty[b], (uint32_t)((i >> 1) - 1) & 1u, p.wait_ns)) {
          flags[0] = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)b * p.acc_cols;
        const int kb0 = (int)((long)sp * p.num_kb / p.splits), kb1 = (int)((long)(sp + 1) * p.num_kb / p.splits);
        #pragma unroll 1
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int s = it % S;
          if (!mbar_wait(&full[s], (uint32_t)(it / S) & 1u, p.wait_ns)) {
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
    if constexpr (DSM) cluster_arrive_release();
  } else {
    // epilogue warps 2..5: TMEM lane quarter q = warp % 4, tile row r
    const int q = warp & 3;
    const int r = q * 32 + lane;
    int ebuf = 0;   // TMA output box in use
    int tn, tm, sp;
    for (int i = 0; work_item(p, i, tn, tm, sp); ++i) {
      const int b = i & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[b], (uint32_t)(i >> 1) & 1u, p.wait_ns));
      if constexpr (DSM) {
        // past this barrier every CTA of the cluster has finished its MMAs
        // (its operand ring may be overwritten) and armed its receive barrier;
        // every thread arrives exactly once, whatever happened before
        cluster_arrive_release();
        cluster_wait_acquire();
      }
      if (!ok) {
        if (lane == 0) flags[0] = 1;
        break;
      }
      tc_fence_after();
      const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)b * p.acc_cols;
      const int m_base = tm * BN;
      const int n = tn * TC_BM + r;
      const float brow = (p.bias && n < p.N) ? p.bias[n] : 0.f;
      if constexpr (RED == RED_NONE) {
        // 16-token chunks; the TMEM load of chunk c+1 is in flight while chunk
        // c goes out
        uint32_t nxt[16];
        tmem_ld16_async(trow, nxt);
        tmem_wait_ld();
        tmem_reg_fence16(nxt);
        #pragma unroll 1
        for (int c0 = 0; c0 < BN; c0 += 16) {
          float v[16];
#pragma unroll
          for (int k = 0; k < 16; ++k) v[k] = __uint_as_float(nxt[k]);
          const bool more = c0 + 16 < BN;
          if (more) {
            tmem_ld16_async(trow + c0 + 16, nxt);
          } else {   // accumulator drained: the MMA warp may reuse it
            tc_fence_before();
            mbar_arrive(&acc_empty[b]);
          }
          if constexpr (TMA_OUT) epilogue_tma<EK>(p, &tmO, tn, m_base + c0, r, v, brow, stg_raw, xch, ebuf);
          else epilogue_chunk(p, tn, m_base + c0, 16, r, v, stage);
          if (more) {
            tmem_wait_ld();
            tmem_reg_fence16(nxt);
          }
        }
      } else if constexpr (RED == RED_DSMEM) {
        // token slice q of this split's partial goes to rank q (= split q) of
        // the cluster in bf16, two rows per 16-byte message: the lanes of rows
        // r and r+1 swap halves of their packed 4-token groups 2k and 2k+1,
        // so that the even lane sends group 2k of both rows and the odd lane
        // group 2k+1; group g of the slice for row pair r/2 lands at
        // [sp][g][r/2] there
        const int ngs = cpr / 4;
        const bool odd = lane & 1;
        const uint32_t rcv0 = smem_u32(smem + p.rcv_off) + (uint32_t)(sp * ngs * 64 + (r >> 1)) * 16u;
        const uint32_t bar0 = smem_u32(rcv_bar);
        // destination rank and group of this lane's next message (group 2k + odd)
        int dst = (odd && ngs == 1) ? 1 : 0, gl = (odd && ngs > 1) ? 1 : 0;
        #pragma unroll 1
        for (int c0 = 0; c0 < BN; c0 += 64) {   // up to four TMEM loads in flight, one wait
          const int nq = min(4, (BN - c0) / 16);   // BN is a multiple of 16
          uint32_t raw[64];
#pragma unroll
          for (int qq = 0; qq < 4; ++qq)
            if (qq < nq) tmem_ld16_async(trow + c0 + 16 * qq, raw + 16 * qq);
          tmem_wait_ld();
#pragma unroll
          for (int qq = 0; qq < 4; ++qq) tmem_reg_fence16(raw + 16 * qq);
          for_upto<8, 2>(2 * nq, [&](int k) {
            const uint32_t* a = raw + 8 * k;
            const uint32_t p0 = pack_bf16x2(__uint_as_float(a[0]), __uint_as_float(a[1]));
            const uint32_t p1 = pack_bf16x2(__uint_as_float(a[2]), __uint_as_float(a[3]));
            const uint32_t p2 = pack_bf16x2(__uint_as_float(a[4]), __uint_as_float(a[5]));
            const uint32_t p3 = pack_bf16x2(__uint_as_float(a[6]), __uint_as_float(a[7]));
            const uint32_t got0 = __shfl_xor_sync(0xffffffffu, odd ? p0 : p2, 1);
            const uint32_t got1 = __shfl_xor_sync(0xffffffffu, odd ? p1 : p3, 1);
            const uint4 w = odd ? make_uint4(got0, got1, p2, p3) : make_uint4(p0, p1, got0, got1);
            st_async_u4(mapa_shared(rcv0 + (uint32_t)gl * 1024u, (uint32_t)dst), w, mapa_shared(bar0, (uint32_t)dst));
            // two groups on: a select per rank boundary, not a branch
            gl += 2;
            bool wrap = gl >= ngs;
            gl = wrap ? gl - ngs : gl;
            dst += wrap ? 1 : 0;
            wrap = gl >= ngs;
            gl = wrap ? gl - ngs : gl;
            dst += wrap ? 1 : 0;
          });
        }
      } else if constexpr (RED == RED_DSMEM32) {
        // token slice q of this split's partial goes to rank q (= split q) of
        // the cluster: float4 group g of the slice lands at [sp][g][r] there
        const int ngs = cpr / 4;
        const uint32_t rcv0 = smem_u32(smem + p.rcv_off) + (uint32_t)(sp * ngs * TC_BM + r) * 16u;
        const uint32_t bar0 = smem_u32(rcv_bar);
        int dst = 0, gl = 0;   // destination rank and group of the next float4
        #pragma unroll 1
        for (int c0 = 0; c0 < BN; c0 += 64) {   // up to four TMEM loads in flight, one wait
          const int nq = min(4, (BN - c0) / 16);   // BN is a multiple of 16
          uint32_t raw[64];
#pragma unroll
          for (int qq = 0; qq < 4; ++qq)
            if (qq < nq) tmem_ld16_async(trow + c0 + 16 * qq, raw + 16 * qq);
          tmem_wait_ld();
#pragma unroll
          for (int qq = 0; qq < 4; ++qq) tmem_reg_fence16(raw + 16 * qq);
          for_upto<16>(4 * nq, [&](int qq) {
            st_async_f4(mapa_shared(rcv0 + (uint32_t)gl * (TC_BM * 16), (uint32_t)dst),
                        make_float4(__uint_as_float(raw[4 * qq]), __uint_as_float(raw[4 * qq + 1]),
                                    __uint_as_float(raw[4 * qq + 2]), __uint_as_float(raw[4 * qq + 3])),
                        mapa_shared(bar0, (uint32_t)dst));
            const bool wrap = ++gl == ngs;   // next rank: a select, not a branch
            gl = wrap ? 0 : gl;
            dst += wrap ? 1 : 0;
          });
        }
      } else if constexpr (RED == RED_L2_CLUSTER) {
        // this split's fp32 partial to the workspace as [col/4][row][4]: each
        // thread stores float4 of 4 consecutive columns, a warp one 512-byte run
        const size_t cl = (size_t)tm * gridDim.x + tn;
        float* w = p.ws + ((cl * p.splits + sp) * (size_t)(BN / 4)) * (TC_BM * 4) + (size_t)r * 4;
        #pragma unroll 1
        for (int c0 = 0; c0 < BN; c0 += 64) {   // up to four TMEM loads in flight, one wait
          const int nq = min(4, (BN - c0) / 16);   // BN is a multiple of 16
          uint32_t raw[64];
#pragma unroll
          for (int qq = 0; qq < 4; ++qq)
            if (qq < nq) tmem_ld16_async(trow + c0 + 16 * qq, raw + 16 * qq);
          tmem_wait_ld();
#pragma unroll
          for (int qq = 0; qq < 4; ++qq) tmem_reg_fence16(raw + 16 * qq);
#pragma unroll
          for (int qq = 0; qq < 16; ++qq)
            if (qq < 4 * nq)
              __stcg((float4*)(w + (size_t)(c0 / 4 + qq) * (TC_BM * 4)),
                     make_float4(__uint_as_float(raw[4 * qq]), __uint_as_float(raw[4 * qq + 1]),
                                 __uint_as_float(raw[4 * qq + 2]), __uint_as_float(raw[4 * qq + 3])));
        }
        __threadfence();
      } else {
        // workspace mode: [split][tile][col][row] partials, last arrival reduces
        const int tiles = gridDim.x * gridDim.y;
        const int tile_id = tm * gridDim.x + tn;
        #pragma unroll 1
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
          #pragma unroll 1
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
    // every TMA output box has been read out of shared memory (the grid's
    // completion makes the writes visible to the dependent launch)
    if (TMA_OUT && threadIdx.x == 64) bulk_wait_read<0>();
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
  if constexpr (DSM) {
    // Rank q sums its slice of tokens [q*cpr, (q+1)*cpr) over the splits in
    // order once every split's bytes have arrived (the wait also keeps this
    // CTA alive until no store into its shared memory is in flight), then
    // sends the whole slice out as one box.  (When the partials overlay the
    // output boxes, epilogue_tma passes a barrier of all 128 threads before it
    // writes over what was just read.)
    if (warp >= 2) {
      const int r = (warp & 3) * 32 + lane;
      const bool ok = __all_sync(0xffffffffu, mbar_wait_cluster(rcv_bar, 0, p.wait_ns));
      if (!ok) {
        if (lane == 0) raise_error(p.err, ERR_TIMEOUT);
      } else {
        const int n = tn0 * TC_BM + r;
        const float brow = (p.bias && n < p.N) ? p.bias[n] : 0.f;
        float v[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) v[k] = 0.f;
        if constexpr (RED == RED_DSMEM) {
          const uint2* b0 = (const uint2*)(smem + p.rcv_off) + 2 * (r >> 1) + (r & 1);
          switch (cpr / 4) {
            case 1: reduce_slice_smem<1>(b0, p.splits, v); break;
            case 2: reduce_slice_smem<2>(b0, p.splits, v); break;
            case 3: reduce_slice_smem<3>(b0, p.splits, v); break;
            case 4: reduce_slice_smem<4>(b0, p.splits, v); break;
            case 5: reduce_slice_smem<5>(b0, p.splits, v); break;
            case 6: reduce_slice_smem<6>(b0, p.splits, v); break;
            case 7: reduce_slice_smem<7>(b0, p.splits, v); break;
            default: reduce_slice_smem<8>(b0, p.splits, v); break;
          }
        } else {
          const float4* b0 = (const float4*)(smem + p.rcv_off) + r;
          switch (cpr / 4) {
            case 1: reduce_slice_smem<1>(b0, p.splits, v); break;
            case 2: reduce_slice_smem<2>(b0, p.splits, v); break;
            case 3: reduce_slice_smem<3>(b0, p.splits, v); break;
            case 4: reduce_slice_smem<4>(b0, p.splits, v); break;
            case 5: reduce_slice_smem<5>(b0, p.splits, v); break;
            case 6: reduce_slice_smem<6>(b0, p.splits, v); break;
            case 7: reduce_slice_smem<7>(b0, p.splits, v); break;
            default: reduce_slice_smem<8>(b0, p.splits, v); break;
          }
        }
        int ebuf = 0;
        if constexpr (TMA_OUT) epilogue_tma<EK, 32>(p, &tmO, tn0, tm0 * BN + sp0 * cpr, r, v, brow, stg_raw, xch, ebuf);
        if (threadIdx.x == 64) bulk_wait_read<0>();
      }
    }
  }
  if constexpr (RED == RED_L2_CLUSTER) {
    // Every split of this tile has written its partial; the cluster barrier
    // (release / acquire) makes them visible.  Rank q sums columns
    // [q*BN/S, (q+1)*BN/S) over the splits in order and applies the epilogue.
    cluster_sync();
    if (warp >= 2) {
      const int r = (warp & 3) * 32 + lane;
      const int Sp = p.splits;
      const int rank = (int)cluster_ctarank();
      const size_t cl = (size_t)tm0 * gridDim.x + tn0;
      const float* base = p.ws + (cl * Sp * (size_t)(BN / 4) + rank * cpr / 4) * (TC_BM * 4) + (size_t)r * 4;
      const size_t sstride = (size_t)(BN / 4) * (TC_BM * 4);
      const int n = tn0 * TC_BM + r;
      const float brow = (p.bias && n < p.N) ? p.bias[n] : 0.f;
      int ebuf = 0;
      // a slice that would take three or more 4- or 8-token chunks goes out
      // whole: one L2 round trip, one output box
      const bool whole = TMA_OUT && cpr <= 32 && cpr > 8 && cpr % 16 != 0;
      if (whole) {
        float v[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) v[k] = 0.f;
        switch (cpr / 4) {
          case 1: reduce_slice_l2<1>(base, Sp, sstride, v); break;
          case 2: reduce_slice_l2<2>(base, Sp, sstride, v); break;
          case 3: reduce_slice_l2<3>(base, Sp, sstride, v); break;
          case 4: reduce_slice_l2<4>(base, Sp, sstride, v); break;
          case 5: reduce_slice_l2<5>(base, Sp, sstride, v); break;
          case 6: reduce_slice_l2<6>(base, Sp, sstride, v); break;
          case 7: reduce_slice_l2<7>(base, Sp, sstride, v); break;
          default: reduce_slice_l2<8>(base, Sp, sstride, v); break;
        }
        if constexpr (TMA_OUT) epilogue_tma<EK, 32>(p, &tmO, tn0, tm0 * BN + rank * cpr, r, v, brow, stg_raw, xch, ebuf);
      }
      #pragma unroll 1
      for (int cc = 0; !whole && cc < cpr; cc += p.box_m) {
        const int nc = p.box_m;
        float v[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = 0.f;
        const float* b0 = base + (size_t)(cc / 4) * (TC_BM * 4);
        if (nc == 16) reduce_splits_l2<4>(b0, Sp, sstride, v);
        else if (nc == 8) reduce_splits_l2<2>(b0, Sp, sstride, v);
        else reduce_splits_l2<1>(b0, Sp, sstride, v);
        const int m0 = tm0 * BN + rank * cpr + cc;
        if constexpr (TMA_OUT) epilogue_tma<EK>(p, &tmO, tn0, m0, r, v, brow, stg_raw, xch, ebuf);
        else epilogue_chunk(p, tn0, m0, nc, r, v, stage);
      }
      if (TMA_OUT && threadIdx.x == 64) bulk_wait_read<0>();
    }
  }
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols) : "memory");
  }
}


// ---------------------------------------------------------------------------
// Two-SM GEMM (persistent, many tiles): a pair of CTAs (a cluster of 2) runs
// one M = 256 MMA per K step -- A = 256 weight rows, 128 in each CTA's shared
// memory, B = BN tokens, BN / 2 in each -- and each CTA's TMEM accumulates its
// own 128 rows for all BN tokens.  Per K step an SM then streams 128 + BN/2
// operand rows through TMA and the MMA instead of 128 + BN, which is what
// bounds the one-SM tile's main loop.  The even CTA's thread issues the MMAs
// and owns the stage barriers: both CTAs load their halves into their own
// shared memory and count the bytes on the even CTA's `full` barrier; the
// MMA completion is multicast to both CTAs' `empty` / `acc_full` barriers;
// both CTAs run the epilogue of their own rows, whose drained accumulators
// the even CTA's `acc_empty` counts (256 arrivals).
template <int EK>
__global__ void __launch_bounds__(TC_PAIR_THREADS, 1)
    tc_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                        const __grid_constant__ CUtensorMap tmO, TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned; derived from smem_raw by pointer arithmetic so that the
  // compiler keeps it (and everything indexed from it) in the shared window
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int BN = p.bn, BNh = BN / 2, S = p.stages;
  const uint32_t bh_bytes = (uint32_t)BNh * TC_BK * 2;
  const uint32_t stage_tx = 2u * (TC_A_BYTES + bh_bytes);   // both CTAs' halves of a stage
  uint8_t* a_s = smem;
  uint8_t* b_s = smem + (size_t)S * TC_A_BYTES;
  uint8_t* stg_raw = smem + p.stg_off;
  float* xch = (float*)(smem + p.xch_off);
  uint64_t* full = (uint64_t*)(smem + p.bar_off);   // the even CTA's count both halves
  uint64_t* empty = full + S;
  uint64_t* acc_full = empty + S;      // [2]
  uint64_t* acc_empty = acc_full + 2;  // [2] the even CTA's: 512 arrivals (256 epilogue threads per CTA)
  uint32_t* tmem_slot = (uint32_t*)(acc_empty + 2);
  int* flags = (int*)(tmem_slot + 1);  // [0] abort, [2] stages issued, [3] stages consumed

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int pair = (int)(blockIdx.x >> 1), npairs = (int)(gridDim.x >> 1);
  const uint32_t ncols = 2 * p.acc_cols;
  // work item i of this pair: pair tile pair + i * npairs = (256-row block tn2, token tile tm)
  auto item = [&](int i, int& tn2, int& tm) -> bool {
    const int t = pair + i * npairs;
    if (t >= p.num_tiles) return false;
    tm = t % p.tiles_m;
    tn2 = t / p.tiles_m;
    return true;
  };
  int tn0 = 0, tm0 = 0;
  const bool has_work = item(0, tn0, tm0);
  const int npre = has_work ? min(S, p.num_kb) : 0;
  constexpr bool TMA_OUT = EK != EK_GENERIC;
  static_assert(TMA_OUT, "the pair kernel stores through TMA boxes");

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 512);
    }
    flags[0] = flags[1] = flags[2] = flags[3] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // both CTAs' barriers exist before either signals the other's
  cluster_sync();
  const uint32_t full0 = mapa_shared(smem_u32(full), 0);          // the even CTA's full[0]
  const uint32_t acc_empty0 = mapa_shared(smem_u32(acc_empty), 0);
  uint64_t pol_w = 0, pol_x = 0;
  if (threadIdx.x == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(&tmW) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(&tmX) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(&tmO) : "memory");
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol_w));
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol_x));
  }
  // the first stages' weight halves, before the wait on the previous kernel
  // (after it, for a launch that may be skipped at run time)
  auto issue_weight_prologue = [&]() {
    for (int i = 0; i < npre; ++i) {
      if (leader) mbar_expect_tx(&full[i], stage_tx);
      tma_load_2d_pair(&tmW, full0 + 8u * (uint32_t)i, a_s + (size_t)i * TC_A_BYTES, i * TC_BK,
                       (2 * tn0 + (int)rank) * TC_BM, pol_w);
    }
  };
  if (threadIdx.x == 0 && !p.skip) issue_weight_prologue();
  pdl_wait();
  if (p.skip) {
    // nothing has been issued yet and the flag is the same for both CTAs of
    // the pair: they leave together, with no copy or arrival in flight
    if (*p.skip) return;
    if (threadIdx.x == 0) issue_weight_prologue();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  cta_sync();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {   // producer (both CTAs): this CTA's A rows and B half of each stage
      int it = 0;
      bool ok = true;
      int tn2, tm;
      for (int i = 0; ok && item(i, tn2, tm); ++i) {
        for (int kb = 0; kb < p.num_kb; ++kb, ++it) {
          const int s = it % S;
          const uint32_t fb = full0 + 8u * (uint32_t)s;
          if (it < npre) {   // weight half already in flight
            tma_load_2d_pair(&tmX, fb, b_s + (size_t)s * bh_bytes, kb * TC_BK, tm * BN + (int)rank * BNh, pol_x);
            continue;
          }
          if (!mbar_wait(&empty[s], ((uint32_t)(it / S) & 1u) ^ 1u)) {
            flags[0] = 1;
            ok = false;
            break;
          }
          if (leader) mbar_expect_tx(&full[s], stage_tx);
          tma_load_2d_pair(&tmW, fb, a_s + (size_t)s * TC_A_BYTES, kb * TC_BK, (2 * tn2 + (int)rank) * TC_BM, pol_w);
          tma_load_2d_pair(&tmX, fb, b_s + (size_t)s * bh_bytes, kb * TC_BK, tm * BN + (int)rank * BNh, pol_x);
        }
      }
      flags[2] = it;
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && leader) {   // MMA issuer: the even CTA only
      const uint32_t idesc = idesc_bf16(2 * TC_BM, BN);
      int it = 0;
      bool ok = true;
      int tn2, tm;
      for (int i = 0; ok && item(i, tn2, tm); ++i) {
        const int b = i & 1;
        // both CTAs' epilogues must have drained the accumulator of item i - 2
        if (i >= 2 && !mbar_wait(&acc_empty[b], (uint32_t)((i >> 1) - 1) & 1u)) {
          flags[0] = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)b * p.acc_cols;
        for (int kb = 0; kb < p.num_kb; ++kb, ++it) {
          const int s = it % S;
          if (!mbar_wait(&full[s], (uint32_t)(it / S) & 1u)) {
            flags[0] = 1;
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = sw128_desc(smem_u32(a_s + (size_t)s * TC_A_BYTES));
          const uint64_t bd = sw128_desc(smem_u32(b_s + (size_t)s * bh_bytes));
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k) umma_bf16_pair(d, ad + 2 * k, bd + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          umma_commit_pair_mc(&empty[s], 3);   // both CTAs' halves of the stage are free
        }
        if (ok) umma_commit_pair_mc(&acc_full[b], 3);
      }
      flags[3] = it;
    }
    __syncwarp();
  } else {
    // epilogue warps 2..9 of both CTAs: TMEM lane quarter q, this CTA's tile
    // row r; set 0 (warps 2..5) takes the 32-token chunks 0, 2, 4, ..., set 1
    // (warps 6..9) chunks 1, 3, 5, ..., each with its own boxes and barrier
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const int set = warp >= 6 ? 1 : 0;
    uint8_t* sboxes = stg_raw + (size_t)set * p.set_bytes;
    float* sxch = (float*)((uint8_t*)xch + (size_t)set * p.set_bytes);
    int ebuf = 0;
    int tn2, tm;
    for (int i = 0; item(i, tn2, tm); ++i) {
      const int b = i & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[b], (uint32_t)(i >> 1) & 1u));
      if (!ok) {
        if (lane == 0) flags[0] = 1;
        break;
      }
      tc_fence_after();
      const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)b * p.acc_cols;
      const int tile_n = 2 * tn2 + (int)rank;   // this CTA's 128-row block
      const int m_base = tm * BN;
      const int n = tile_n * TC_BM + r;
      const float brow = (p.bias && n < p.N) ? p.bias[n] : 0.f;
      // 32-token chunks (BN is a multiple of 32, at least 128): this set's
      // every other chunk, the next one's TMEM load in flight meanwhile
      uint32_t nxt[32];
      const int cf = 32 * set;
      tmem_ld32_async(trow + cf, nxt);
      tmem_wait_ld();
      tmem_reg_fence16(nxt);
      tmem_reg_fence16(nxt + 16);
      for (int c0 = cf; c0 < BN; c0 += 64) {
        float v[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) v[k] = __uint_as_float(nxt[k]);
        const bool more = c0 + 64 < BN;
        if (more) {
          tmem_ld32_async(trow + c0 + 64, nxt);
        } else {   // this thread is done with the accumulator: tell the MMA issuer
          tc_fence_before();
          mbar_arrive_remote(acc_empty0 + 8u * (uint32_t)b);
        }
        epilogue_tma<EK, 32>(p, &tmO, tile_n, m_base + c0, r, v, brow, sboxes, sxch, ebuf);
        if (more) {
          tmem_wait_ld();
          tmem_reg_fence16(nxt);
          tmem_reg_fence16(nxt + 16);
        }
      }
    }
    if (threadIdx.x == 64 + 128 * set) bulk_wait_read<0>();   // this set's boxes have been read out
  }
  tc_fence_before();
  cta_sync();
  if (flags[0]) {
    // unwind: the even CTA waits (bounded) for stages issued but never consumed
    if (threadIdx.x == 0) {
      if (leader)
        for (int i = flags[3]; i < flags[2]; ++i) mbar_wait(&full[i % S], (uint32_t)(i / S) & 1u);
      raise_error(p.err, ERR_TIMEOUT);
    }
    cta_sync();
  }
  // neither CTA leaves while the other may still signal its barriers or
  // (through the MMA) read its shared memory
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols) : "memory");
  }
}

using TcKernel = void (*)(CUtensorMap, CUtensorMap, CUtensorMap, TcParams);

TcKernel tc_pair_kernel(int ek) {
  switch (ek) {
    case EK_F32: return tc_gemm_pair_kernel<EK_F32>;
    case EK_BF16: return tc_gemm_pair_kernel<EK_BF16>;
    case EK_ADD: return tc_gemm_pair_kernel<EK_ADD>;
    case EK_GEGLU: return tc_gemm_pair_kernel<EK_GEGLU>;
    default: return nullptr;
  }
}

// The instantiation for a reduction mode and epilogue kind (nullptr where the
// pair cannot occur: the workspace mode stores from the threads, the
// shared-memory exchange needs TMA outputs).
TcKernel tc_kernel(int red, int ek) {
#define RAVEL_TC_K(R, E) \
  if (red == R && ek == E) return tc_gemm_kernel<R, E>;
  RAVEL_TC_K(RED_NONE, EK_F32) RAVEL_TC_K(RED_NONE, EK_BF16) RAVEL_TC_K(RED_NONE, EK_ADD)
  RAVEL_TC_K(RED_NONE, EK_GEGLU) RAVEL_TC_K(RED_NONE, EK_GENERIC)
  RAVEL_TC_K(RED_L2_CLUSTER, EK_TMA_ANY) RAVEL_TC_K(RED_L2_CLUSTER, EK_GENERIC)
  RAVEL_TC_K(RED_DSMEM, EK_TMA_ANY) RAVEL_TC_K(RED_DSMEM32, EK_TMA_ANY)
  RAVEL_TC_K(RED_WORKSPACE, EK_GENERIC)
#undef RAVEL_TC_K
  return nullptr;
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

// 3D map over a row-major bf16 [rows][cols] matrix (cols a multiple of 64)
// viewed as (64 elements, rows, cols / 64 k-tiles): a box of box_rows x nkb
// lands as nkb consecutive K-major 128-byte-swizzled tiles of box_rows rows.
cudaError_t encode_kt(CUtensorMap* m, const void* base, int rows, int cols, int ld, int box_rows, int nkb) {
  cuuint64_t dims[3] = {(cuuint64_t)TC_BK, (cuuint64_t)rows, (cuuint64_t)(cols / TC_BK)};
  cuuint64_t strides[2] = {(cuuint64_t)ld * 2, (cuuint64_t)TC_BK * 2};
  cuuint32_t box[3] = {(cuuint32_t)TC_BK, (cuuint32_t)box_rows, (cuuint32_t)nkb};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// 2D map over a row-major output [rows][cols] (row stride ld elements) for
// TMA stores: box = box_cols x box_rows, no swizzle (the box is dense in
// shared memory), writes past the extents clipped.
cudaError_t encode_out(CUtensorMap* m, void* base, int rows, int cols, int ld, bool bf, int box_cols, int box_rows) {
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * (bf ? 2 : 4)};
  cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, bf ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                        CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Token-tile width: up to 128 tokens, the smallest of 32, 48, .., 128 (the
// MMA's N steps by 16) that holds M; beyond 128 tokens, the multiple of 16 in
// [128, 256] whose tile count fills whole waves of the SMs best (per-CTA work
// ~ waves x BN), larger BN on ties.
int pick_bn(int M, int tiles_n, int num_sms) {
  if (M <= 128) return std::max(32, (M + 15) / 16 * 16);
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
std::atomic<int> g_withhold{0};   // launches left to run with a withheld arrival (fault injection)
constexpr unsigned long long kWithholdWaitNs = 2000000ull;   // their wait limit: 2 ms
bool g_pair_gemm = true;  // persistent launches of many tiles on SM pairs
int g_pair_bn_max = 256;  // widest token tile of a pair launch

// Two-SM launch of a persistent GEMM (see tc_gemm_pair_kernel): token-tile
// width BN (a multiple of 32 in [128, 256]) minimising waves x (BN + 64) --
// the work of a pair's tiles plus a fixed cost per tile of about 64 token
// columns (accumulator hand-off and epilogue pipeline, ~1 us) -- larger BN on
// ties; then the usual TMA epilogue layout.
int pick_bn_pair(int M, int tiles_n2, int slots) {
  int bn = 256;
  long best = -1;
  for (int c = g_pair_bn_max; c >= 128; c -= 32) {
    const long tiles = (long)tiles_n2 * ((M + c - 1) / c);
    const long cost = (tiles + slots - 1) / slots * (c + 64);
    if (best < 0 || cost < best) {
      best = cost;
      bn = c;
    }
  }
  return bn;
}

cudaError_t launch_gemm_pair(const GemmArgs& g, const TcWorkspace& ws, int num_sms, cudaStream_t st, int ek,
                             bool out_bf, int es) {
  const int tiles_n = (g.N + TC_BM - 1) / TC_BM;
  const int tiles_n2 = (g.N + 2 * TC_BM - 1) / (2 * TC_BM);
  const int slots = num_sms / 2;
  const int bn = pick_bn_pair(g.M, tiles_n2, slots);
  const int tiles_m = (g.M + bn - 1) / bn;
  const int num_tiles = tiles_n2 * tiles_m;
  const int num_kb = (g.K + TC_BK - 1) / TC_BK;
  uint32_t acc_cols = 32;
  while ((int)acc_cols < bn) acc_cols <<= 1;
  const int box_m = 32;
  const uint32_t box_bytes =
      (uint32_t)(((size_t)box_m * (g.epi == EPI_GEGLU ? 64 : TC_BM) * es + 1023) / 1024 * 1024);
  const size_t stg_bytes = 2 * (size_t)box_bytes;
  const size_t xch_bytes = g.epi == EPI_GEGLU ? (XCH_BYTES + 1023) / 1024 * 1024 : 0;
  // each of the two epilogue warp sets has its own boxes and exchange tile
  const size_t set_bytes = stg_bytes + xch_bytes;
  const size_t fixed = 1024 + 2 * set_bytes + 256;
  const int stage_bytes = TC_A_BYTES + (bn / 2) * TC_BK * 2;
  const int stages = std::min(8, (int)((TC_SMEM_MAX - fixed) / stage_bytes));
  if (stages < 2) return cudaErrorInvalidConfiguration;
  const size_t ring = ((size_t)stages * stage_bytes + 1023) / 1024 * 1024;
  const uint32_t stg_off = (uint32_t)ring;
  const uint32_t xch_off = stg_off + (uint32_t)stg_bytes;
  const uint32_t bar_off = stg_off + 2 * (uint32_t)set_bytes;
  const size_t smem = 1024 + bar_off + (size_t)(2 * stages + 4) * 8 + 4 + 16 + 64;
  if (smem > (size_t)TC_SMEM_MAX) return cudaErrorInvalidConfiguration;
  CUtensorMap mw, mx, mo;
  cudaError_t e = encode_2d(&mw, g.W, g.N, g.K, g.ldw, TC_BM);
  if (e == cudaSuccess) e = encode_2d(&mx, g.A, g.M, g.K, g.lda, bn / 2);
  if (e == cudaSuccess)
    e = encode_out(&mo, g.out, g.M, g.epi == EPI_GEGLU ? g.N / 2 : g.N, g.ldo, out_bf,
                   g.epi == EPI_GEGLU ? 64 : TC_BM, box_m);
  if (e != cudaSuccess) return e;
  TcParams p{g.M, g.N, g.K, bn, stages, 1, num_kb, RED_NONE, (uint32_t)ring, acc_cols, tiles_n, tiles_m, num_tiles,
             (int)g.epi, g.out_dt == DT_BF16 ? 1 : 0, g.out, g.ldo, g.bias, ws.ws, ws.counters, ws.err,
             1, 0, box_m, box_bytes, stg_off, xch_off, 0, bar_off, kTcTimeoutNs, 0, g.skip};
  p.set_bytes = (uint32_t)set_bytes;
  const int npairs = std::min(num_tiles, slots);
  return launch_kernel_cluster(tc_pair_kernel(ek), dim3(2 * npairs), dim3(TC_PAIR_THREADS), smem, st, dim3(2, 1, 1),
                               mw, mx, mo, p);
}

}  // namespace

void debug_withhold_gemm(int launches) { g_withhold.store(launches > 0 ? launches : 0); }

cudaError_t init_tc_gemm() {
  cudaError_t e = get_encoder();
  if (e != cudaSuccess) return e;
  std::vector<const void*> kernels;
  for (int red = 0; red < 5; ++red)
    for (int ek = 0; ek <= EK_TMA_ANY; ++ek)
      if (TcKernel k = tc_kernel(red, ek)) kernels.push_back((const void*)k);
  for (int ek = 0; ek < EK_GENERIC; ++ek) kernels.push_back((const void*)tc_pair_kernel(ek));
  for (const void* k : kernels) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, TC_SMEM_MAX);
    if (e != cudaSuccess) return e;
  }
  // clusters of 16 are beyond the portable limit: use them only if allowed
  bool big = true;
  for (const void* k : kernels) big = big && cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
  if (big) {
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
    if (cudaOccupancyMaxActiveClusters(&n, tc_kernel(RED_L2_CLUSTER, EK_GENERIC), &cfg) == cudaSuccess && n > 0)
      g_max_cluster = 16;
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
  if (g.max_splits > 0) splits = std::min(splits, g.max_splits);
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
  int reduce = splits == 1 ? RED_NONE : (cluster ? RED_L2_CLUSTER : RED_WORKSPACE);
  {
    // two-SM tiles for a persistent launch whose pair tiles fill at least
    // three quarters of the pairs of SMs
    const bool obf = g.epi == EPI_GEGLU || (g.epi != EPI_ADD_F32 && g.out_dt == DT_BF16);
    const int oes = obf ? 2 : 4;
    const bool aligned = ((uintptr_t)g.out & 15) == 0 && ((size_t)g.ldo * oes) % 16 == 0;
    const int tn2 = (g.N + 2 * TC_BM - 1) / (2 * TC_BM), slots = num_sms / 2;
    const int pbn = pick_bn_pair(g.M, tn2, slots);
    const long pair_tiles = (long)tn2 * ((g.M + pbn - 1) / pbn);
    if (cluster && g_pair_gemm && splits == 1 && aligned && 4 * pair_tiles >= 3 * slots) {
      const int ek = g.epi == EPI_GEGLU ? EK_GEGLU : g.epi == EPI_ADD_F32 ? EK_ADD : obf ? EK_BF16 : EK_F32;
      return launch_gemm_pair(g, ws, num_sms, st, ek, obf, oes);
    }
  }
  const int cpr = bn / splits;   // a multiple of 4 whenever the splits form a cluster
  uint32_t acc_cols = 32;
  while ((int)acc_cols < bn) acc_cols <<= 1;
  const int stage_bytes = TC_A_BYTES + bn * TC_BK * 2;
  const int kb_per_item = (num_kb + splits - 1) / splits;
  const int grid_ctas = splits > 1 ? tiles * splits : std::min(tiles, num_sms);
  const int items = splits > 1 ? 1 : (tiles + grid_ctas - 1) / grid_ctas;
  int stages = std::min(8, TC_SMEM_BUDGET / stage_bytes);
  // a split-K launch is latency-bound: enough stages for its whole (short) K
  // range when that fits, so that no operand load waits for a freed stage
  if (splits > 1) stages = std::min(stages, std::max(2, TC_RING_SPLIT / stage_bytes));
  stages = std::max(2, std::min(stages, std::max(2, kb_per_item * items)));
  // one-shot: a cluster split whose whole K range fits a ring of up to 200 KB
  // takes its weight and token k-tiles in one box each (K a multiple of 64)
  const bool oneshot = splits > 1 && cluster && g.K % TC_BK == 0 && g.K / TC_BK <= 256 &&
                       (size_t)kb_per_item * stage_bytes <= (size_t)TC_SMEM_BUDGET;
  if (oneshot) stages = kb_per_item;   // the ring is exactly one box deep
  const size_t ring = ((size_t)stages * stage_bytes + 1023) / 1024 * 1024;
  // outputs through TMA boxes when the output rows are 16-byte aligned
  const bool out_bf = g.epi == EPI_GEGLU || (g.epi != EPI_ADD_F32 && g.out_dt == DT_BF16);
  const int es = out_bf ? 2 : 4;
  const bool tma_out = reduce != RED_WORKSPACE && ((uintptr_t)g.out & 15) == 0 && ((size_t)g.ldo * es) % 16 == 0;
  int box_m = 0;
  // partials exchanged in bf16 where the caller allows it, else in fp32
  const bool xbf = g.xbf16 != 0;
  uint32_t box_bytes = 0, stg_off = (uint32_t)ring, xch_off = 0, rcv_off = 0, bar_off = 0;
  size_t smem = 0;
  auto layout = [&](bool dsmem) {
    box_m = splits == 1 ? 16
            : (tma_out && cpr <= 32 && (dsmem || (cpr > 8 && cpr % 16 != 0))) ? cpr   // the whole slice in one box
            : (cpr % 16 == 0 ? 16 : (cpr % 8 == 0 ? 8 : 4));
    box_bytes = (uint32_t)(((size_t)box_m * (g.epi == EPI_GEGLU ? 64 : TC_BM) * es + 1023) / 1024 * 1024);
    const size_t stg_bytes = tma_out ? 2 * (size_t)box_bytes : (STG_BYTES + 1023) / 1024 * 1024;
    const size_t xch_bytes = (tma_out && g.epi == EPI_GEGLU) ? (XCH_BYTES + 1023) / 1024 * 1024 : 0;
    // received partials (all splits' slices of this rank) overlay the operand
    // ring, else the boxes + exchange
    const size_t rcv_bytes = dsmem ? (size_t)TC_BM * bn * (xbf ? 2 : 4) : 0;
    const bool in_ring = rcv_bytes <= ring;
    xch_off = stg_off + (uint32_t)stg_bytes;
    rcv_off = in_ring ? 0u : stg_off;
    bar_off = stg_off + (uint32_t)std::max(stg_bytes + xch_bytes, in_ring ? (size_t)0 : rcv_bytes);
    smem = 1024 + bar_off + (size_t)(2 * stages + 5) * 8 + 4 + 16 + 64;
  };
  // partials by st.async into the owning rank's shared memory when the token
  // slice fits one output box (<= 32 tokens) and the receive area fits
  bool dsmem = reduce == RED_L2_CLUSTER && tma_out && cpr <= 32;
  layout(dsmem);
  if (dsmem && smem > (size_t)TC_SMEM_MAX) {
    dsmem = false;
    layout(false);
  }
  if (dsmem) reduce = xbf ? RED_DSMEM : RED_DSMEM32;
  CUtensorMap mw, mx, mo;
  memset(&mo, 0, sizeof(mo));
  cudaError_t e = oneshot ? encode_kt(&mw, g.W, g.N, g.K, g.ldw, TC_BM, kb_per_item)
                          : encode_2d(&mw, g.W, g.N, g.K, g.ldw, TC_BM);
  if (e == cudaSuccess)
    e = oneshot ? encode_kt(&mx, g.A, g.M, g.K, g.lda, bn, kb_per_item) : encode_2d(&mx, g.A, g.M, g.K, g.lda, bn);
  if (e == cudaSuccess && tma_out)
    e = encode_out(&mo, g.out, g.M, g.epi == EPI_GEGLU ? g.N / 2 : g.N, g.ldo, out_bf,
                   g.epi == EPI_GEGLU ? 64 : TC_BM, box_m);
  if (e != cudaSuccess) return e;
  TcParams p{g.M, g.N, g.K, bn, stages, splits, num_kb, reduce, (uint32_t)ring, acc_cols, tiles_n, tiles_m, tiles,
             (int)g.epi, g.out_dt == DT_BF16 ? 1 : 0, g.out, g.ldo, g.bias, ws.ws, ws.counters, ws.err,
             tma_out ? 1 : 0, oneshot ? 1 : 0, box_m, box_bytes, stg_off, xch_off, rcv_off, bar_off, kTcTimeoutNs, 0,
             g.skip};
  // fault injection (tests): a launch without a cluster may be told to wait
  // for an arrival that never comes, with a short limit
  if ((reduce == RED_NONE || reduce == RED_WORKSPACE) && g_withhold.load() > 0 && g_withhold.fetch_sub(1) > 0) {
    p.withhold = 1;
    p.wait_ns = kWithholdWaitNs;
  }
  const dim3 grid = splits > 1 ? dim3(tiles_n, tiles_m, splits) : dim3(grid_ctas);
  const dim3 block(TC_THREADS);
  // persistent launches: one instantiation per epilogue kind; split-K
  // launches: one for all TMA epilogues
  const int ek = !tma_out ? EK_GENERIC
                 : reduce != RED_NONE ? EK_TMA_ANY
                 : g.epi == EPI_GEGLU ? EK_GEGLU : g.epi == EPI_ADD_F32 ? EK_ADD : out_bf ? EK_BF16 : EK_F32;
  const TcKernel k = tc_kernel(reduce, ek);
  if (!k) return cudaErrorInvalidConfiguration;
  const bool clustered = reduce == RED_L2_CLUSTER || reduce == RED_DSMEM || reduce == RED_DSMEM32;
  return launch_kernel(k, grid, block, smem, st, clustered ? (unsigned)splits : 1u, mw, mx, mo, p);
}

}  // namespace ravel
