// Projection GEMM on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
//   out[m][n] (op)= sum_k X[m][k] * W[n][k]       X: activations [M][K] bf16
//                                                  W: weights     [N][K] bf16 (K-major)
//
// Swap-AB tiling: a CTA owns 128 weight rows (the MMA's M = 128 TMEM lanes)
// and BN tokens (the MMA's N, 16..256): with only 50-66 tokens per robot the
// weights are the large operand, and this keeps one kernel for both the
// bandwidth-bound batch-1 case (BN = 64/96, split-K over the grid) and the
// compute-bound large-batch case (BN = 256 token tiles).
//
// Warp roles (192 threads): warp 0 = TMA producer, warp 1 = TMEM allocator +
// single-thread MMA issuer, warps 2..5 = epilogue (warp w reads TMEM lanes
// 32*(w%4)..+31).  Operand tiles are 64 K-elements wide (one 128-byte
// swizzle row) and sit in an S-stage shared-memory ring guarded by mbarriers.
// Every wait is bounded: on timeout the kernel raises ERR_TIMEOUT in the
// device error word and unwinds instead of hanging.
//
// Split-K: grid.z CTAs share a tile; each writes its fp32 partial to a
// workspace, and the last to arrive (per-tile counter) sums the partials in
// split order (deterministic) and runs the epilogue, then resets the counter.
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
constexpr int TC_SMEM_BUDGET = 200 * 1024;                     // operand ring
constexpr int TC_SMEM_MAX = 227 * 1024;

struct TcParams {
  int M, N, K;
  int bn, stages, splits, num_kb;
  int cluster_reduce;   // the grid.z splits of a tile form a cluster; 1: reduce through DSMEM, 2: through L2
  uint32_t ring_bytes;  // operand ring (also holds the fp32 partial tile in cluster mode)
  int epi;          // Epi value, or EPI_GEGLU
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

// v[i] += sum over splits s = 0..S-1 (in order) of the partial at column
// cc + i of split s; base points at this thread's row of split 0, column 0.
// Up to 64 loads are in flight per batch; splits past S add exact zeros.
template <int NC>
__device__ __forceinline__ void reduce_splits_l2(const float* base, int S, int BN, int cc, float v[16]) {
  constexpr int G = 64 / NC;
  for (int s0 = 0; s0 < S; s0 += G) {
    float x[G][NC];
#pragma unroll
    for (int u = 0; u < G; ++u)
#pragma unroll
      for (int i = 0; i < NC; ++i)
        x[u][i] = (s0 + u < S) ? __ldcg(base + ((size_t)(s0 + u) * BN + cc + i) * 128) : 0.f;
#pragma unroll
    for (int u = 0; u < G; ++u)
#pragma unroll
      for (int i = 0; i < NC; ++i) v[i] += x[u][i];
  }
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Apply the epilogue to nc (<= 16) consecutive tokens m0.. of tile row r.
// `xch` is the 64x16 exchange tile of the GeGLU epilogue (all 128 epilogue
// threads must call this together in that mode).
__device__ __forceinline__ void apply_epilogue(const TcParams& p, int tile_n, int r, int m0, float v[16],
                                               float* xch, int nc = 16) {
  if (p.epi == EPI_GEGLU) {
    // rows 0..63 of the tile are gate features, rows 64..127 the matching up features
    if (r >= 64) {
#pragma unroll
      for (int i = 0; i < 16; ++i) xch[(r - 64) * 17 + i] = v[i];
    }
    epi_bar();
    if (r < 64) {
      const int f = tile_n * 64 + r;
      if (f < p.N / 2) {
        bf16* o = (bf16*)p.out;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int m = m0 + i;
          if (i < nc && m < p.M) o[(size_t)m * p.ldo + f] = __float2bfloat16_rn(gelu_tanh_f(v[i]) * xch[r * 17 + i]);
        }
      }
    }
    epi_bar();
    return;
  }
  const int n = tile_n * TC_BM + r;
  if (n >= p.N) return;
  const float b = p.bias ? p.bias[n] : 0.f;
  if (p.epi == EPI_ADD_F32) {
    // residual accumulate: all loads first, so their latencies overlap
    float* o = (float*)p.out;
    float old[16];
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (i < nc && m0 + i < p.M) old[i] = o[(size_t)(m0 + i) * p.ldo + n];
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (i < nc && m0 + i < p.M) o[(size_t)(m0 + i) * p.ldo + n] = old[i] + (v[i] + b);
    return;
  }
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int m = m0 + i;
    if (i >= nc || m >= p.M) continue;
    float x = v[i] + b;
    const size_t idx = (size_t)m * p.ldo + n;
    {
      if (p.epi == EPI_STORE_SILU) x = silu_f(x);
      if (p.out_bf16)
        ((bf16*)p.out)[idx] = __float2bfloat16_rn(x);
      else
        ((float*)p.out)[idx] = x;
    }
  }
  if (p.vt && n >= p.v_col0) {
    const int g = (n - p.v_col0) / p.vt_hd, d = (n - p.v_col0) % p.vt_hd;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int m = m0 + i;
      if (i >= nc || m >= p.M) continue;
      const int bb = m / p.vt_tokens, kk = m % p.vt_tokens;
      p.vt[((size_t)(bb * p.vt_hkv + g) * p.vt_hd + d) * p.vt_kvp + kk] = __float2bfloat16_rn(v[i] + b);
    }
  }
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
  uint64_t* accb = empty + S;
  uint32_t* tmem_slot = (uint32_t*)(accb + 1);
  int* flags = (int*)(tmem_slot + 1);   // [0] abort, [1] last-split, [2] issued, [3] consumed
  float* xch = (float*)(((uintptr_t)(flags + 4) + 15) & ~(uintptr_t)15);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tile_n = blockIdx.x, tile_m = blockIdx.y, split = blockIdx.z;
  const int kb0 = (int)((long)split * p.num_kb / p.splits);
  const int kb1 = (int)((long)(split + 1) * p.num_kb / p.splits);
  const int nkb = kb1 - kb0;
  uint32_t ncols = 32;
  while ((int)ncols < BN) ncols <<= 1;

  pdl_trigger();
  const int npre = nkb < S ? nkb : S;   // stages whose weight tiles are fetched before the dependency wait
  uint64_t pol_w = 0, pol_x = 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accb, 1);
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
      tma_load_2d(&tmW, &full[i], a_s + (size_t)i * TC_A_BYTES, (kb0 + i) * TC_BK, tile_n * TC_BM, pol_w);
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
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      for (int i = 0; i < npre; ++i)
        tma_load_2d(&tmX, &full[i], b_s + (size_t)i * b_bytes, (kb0 + i) * TC_BK, tile_m * BN, pol_x);
      int i = npre;
      for (; i < nkb; ++i) {
        const int s = i % S;
        const uint32_t ph = (uint32_t)(i / S) & 1u;
        if (!mbar_wait(&empty[s], ph ^ 1u)) {
          flags[0] = 1;
          break;
        }
        mbar_expect_tx(&full[s], TC_A_BYTES + b_bytes);
        const int kx = (kb0 + i) * TC_BK;
        tma_load_2d(&tmW, &full[s], a_s + (size_t)s * TC_A_BYTES, kx, tile_n * TC_BM, pol_w);
        tma_load_2d(&tmX, &full[s], b_s + (size_t)s * b_bytes, kx, tile_m * BN, pol_x);
      }
      flags[2] = i;
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(TC_BM, BN);
      int i = 0;
      for (; i < nkb; ++i) {
        const int s = i % S;
        const uint32_t ph = (uint32_t)(i / S) & 1u;
        if (!mbar_wait(&full[s], ph)) {
          flags[0] = 1;
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint64_t ad = sw128_desc(smem_u32(a_s + (size_t)s * TC_A_BYTES));
        const uint64_t bd = sw128_desc(smem_u32(b_s + (size_t)s * b_bytes));
#pragma unroll
        for (int k = 0; k < TC_BK / 16; ++k)
          umma_bf16(tmem, ad + 2 * k, bd + 2 * k, idesc, (i > 0 || k > 0) ? 1u : 0u);
        umma_commit(&empty[s]);
      }
      flags[3] = i;
      umma_commit(accb);   // arrives once every MMA issued above has completed
    }
    __syncwarp();
  } else {
    // epilogue warps 2..5: TMEM lane quarter q = warp % 4, tile row r
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const bool ok = mbar_wait(accb, 0);
    if (!ok && lane == 0) flags[0] = 1;
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16);
    const int m_base = tile_m * BN;
    if (p.cluster_reduce == 2) {
      // this split's fp32 partial tile to the workspace, column-major per tile
      // ([col][row]) so a warp's stores and the later loads are contiguous
      const size_t cl = (size_t)tile_m * gridDim.x + tile_n;
      float* w = p.ws + ((cl * p.splits + split) * (size_t)BN) * TC_BM + r;
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
#pragma unroll
        for (int i = 0; i < 16; ++i) __stcg(w + (size_t)(c0 + i) * TC_BM, v[i]);
      }
      __threadfence();
    } else if (p.cluster_reduce) {
      // this split's fp32 partial tile into its own shared memory (the drained
      // operand ring), rows padded to BN + 4 floats against bank conflicts
      float* part = (float*)smem;
      const int ld = BN + 4;
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
#pragma unroll
        for (int qq = 0; qq < 4; ++qq)
          *(float4*)(part + (size_t)r * ld + c0 + 4 * qq) = make_float4(v[4 * qq], v[4 * qq + 1], v[4 * qq + 2], v[4 * qq + 3]);
      }
    } else if (p.splits == 1) {
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
        apply_epilogue(p, tile_n, r, m_base + c0, v, xch);
      }
    } else {
      const int tiles = gridDim.x * gridDim.y;
      const int tile_id = tile_m * gridDim.x + tile_n;
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld16(trow + c0, v);
        float* w = p.ws + ((size_t)(split * tiles + tile_id) * BN + c0) * TC_BM + r;
#pragma unroll
        for (int i = 0; i < 16; ++i) __stcg(w + (size_t)i * TC_BM, v[i]);
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
          for (int i = 0; i < 16; ++i) v[i] = 0.f;
          for (int s = 0; s < p.splits; ++s) {
            const float* w = p.ws + ((size_t)(s * tiles + tile_id) * BN + c0) * TC_BM + r;
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] += __ldcg(w + (size_t)i * TC_BM);
          }
          apply_epilogue(p, tile_n, r, m_base + c0, v, xch);
        }
        if (threadIdx.x == 64) p.counters[tile_id] = 0;
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (flags[0]) {
    // unwind: wait (bounded) for the copies this CTA issued but never consumed
    if (threadIdx.x == 0) {
      for (int i = flags[3]; i < flags[2]; ++i) mbar_wait(&full[i % S], (uint32_t)(i / S) & 1u);
      raise_error(p.err, ERR_TIMEOUT);
    }
    __syncthreads();
  }
  if (p.cluster_reduce == 2) {
    // Every split of this tile has written its partial to the workspace; the
    // cluster barrier (release / acquire) makes them visible.  CTA rank q sums
    // columns [q*BN/S, (q+1)*BN/S) over splits 0..S-1 in order (deterministic)
    // with all loads of a chunk in flight together, and applies the epilogue.
    cluster_sync();
    if (warp >= 2) {
      const int r = (warp & 3) * 32 + lane;
      const int S = p.splits;
      const int cpr = BN / S;
      const int rank = (int)cluster_ctarank();
      const size_t cl = (size_t)tile_m * gridDim.x + tile_n;
      const float* base = p.ws + (cl * S * (size_t)BN + rank * cpr) * TC_BM + r;
      for (int cc = 0; cc < cpr; cc += 16) {
        const int nc = min(16, cpr - cc);
        float v[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
        if (nc == 16) reduce_splits_l2<16>(base, S, BN, cc, v);
        else if (nc == 8) reduce_splits_l2<8>(base, S, BN, cc, v);
        else if (nc == 4) reduce_splits_l2<4>(base, S, BN, cc, v);
        else
          for (int i = 0; i < nc; ++i) {
            float one[16] = {};
            reduce_splits_l2<1>(base + (size_t)i * TC_BM, S, BN, cc, one);
            v[i] = one[0];
          }
        apply_epilogue(p, tile_n, r, tile_m * BN + rank * cpr + cc, v, xch, nc);
      }
    }
  } else if (p.cluster_reduce) {
    // Every split of this tile holds its partial in shared memory.  CTA rank q
    // of the cluster sums columns [q*BN/S, (q+1)*BN/S) over ranks 0..S-1 in
    // order (deterministic) through distributed shared memory and applies the
    // epilogue to them.  The second cluster barrier keeps every partial alive
    // until all ranks have read it.
    cluster_sync();
    if (warp >= 2) {
      const int r = (warp & 3) * 32 + lane;
      const int S = p.splits;
      const int cpr = BN / S;
      const int rank = (int)cluster_ctarank();
      const int ld = BN + 4;
      const uint32_t mine = smem_u32((float*)smem + (size_t)r * ld + rank * cpr);
      for (int cc = 0; cc < cpr; cc += 16) {
        const int nc = min(16, cpr - cc);
        float v[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
        // all remote loads of this chunk are in flight together (one DSMEM
        // round trip), then summed in rank order
        if ((nc & 3) == 0) {
          const int n4 = nc >> 2;
          const int rpb = 16 / n4;   // ranks per batch: at most 16 float4 in flight
          for (int s0 = 0; s0 < S; s0 += rpb) {
            float4 x[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const int u = k / n4, qq = k % n4;
              if (s0 + u < S) x[k] = ld_dsmem_f4(mapa_shared(mine + 4u * cc, (uint32_t)(s0 + u)) + 16u * qq);
            }
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const int u = k / n4, qq = k % n4;
              if (s0 + u < S) {
                v[4 * qq] += x[k].x; v[4 * qq + 1] += x[k].y; v[4 * qq + 2] += x[k].z; v[4 * qq + 3] += x[k].w;
              }
            }
          }
        } else {
          // column counts that are not a multiple of 4 (narrow slices): scalar loads
          for (int i0 = 0; i0 < nc; i0 += 4) {
            for (int s0 = 0; s0 < S; s0 += 4) {
              float x[4][4];
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                if (s0 + u >= S) break;
                const uint32_t ra = mapa_shared(mine + 4u * (cc + i0), (uint32_t)(s0 + u));
#pragma unroll
                for (int i = 0; i < 4; ++i)
                  if (i0 + i < nc) x[u][i] = ld_dsmem_f32(ra + 4u * i);
              }
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                if (s0 + u >= S) break;
#pragma unroll
                for (int i = 0; i < 4; ++i)
                  if (i0 + i < nc) v[i0 + i] += x[u][i];
              }
            }
          }
        }
        apply_epilogue(p, tile_n, r, tile_m * BN + rank * cpr + cc, v, xch, nc);
      }
    }
    cluster_sync();
  }
  if (warp == 1) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
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

int pick_bn(int M) {
  const int cands[] = {32, 64, 96, 128};
  for (int c : cands)
    if (M <= c) return c;
  return 256;
}

}  // namespace

int g_max_cluster = 8;   // largest power-of-two cluster the split-K reduction may use

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
  const int bn = pick_bn(g.M);
  const int tiles_n = (g.N + TC_BM - 1) / TC_BM;
  const int tiles_m = (g.M + bn - 1) / bn;
  const int num_kb = (g.K + TC_BK - 1) / TC_BK;
  const int tiles = tiles_n * tiles_m;
  int splits = 1;
  if (tiles < num_sms) splits = std::min(num_kb, std::max(1, num_sms / tiles));
  if (cluster) {
    // the splits of a tile form one cluster: a power of two, at most the cluster
    // limit, whose partials fit the workspace
    int c = 1;
    while (c * 2 <= std::min(splits, g_max_cluster) &&
           (size_t)(c * 2) * tiles * bn * TC_BM * 4 <= ws.ws_bytes)
      c *= 2;
    splits = c;
  } else {
    while (splits > 1 && ((size_t)splits * tiles * bn * TC_BM * 4 > ws.ws_bytes || tiles > ws.n_counters)) --splits;
  }
  const bool cluster_reduce = cluster && splits > 1;
  const int stage_bytes = TC_A_BYTES + bn * TC_BK * 2;
  int stages = std::min(8, TC_SMEM_BUDGET / stage_bytes);
  stages = std::max(2, std::min(stages, std::max(2, (num_kb + splits - 1) / splits)));
  size_t ring = (size_t)stages * stage_bytes;
  if (cluster_reduce) ring = std::max(ring, (size_t)TC_BM * (bn + 4) * 4);
  ring = (ring + 1023) / 1024 * 1024;
  // 1024 alignment slack + ring + barriers / TMEM slot / flags (+ slack) + GeGLU exchange tile
  const size_t smem = 1024 + ring + (2 * stages + 1) * 8 + 128 + 64 * 17 * 4;
  CUtensorMap mw, mx;
  cudaError_t e = encode_2d(&mw, g.W, g.N, g.K, g.ldw, TC_BM);
  if (e == cudaSuccess) e = encode_2d(&mx, g.A, g.M, g.K, g.lda, bn);
  if (e != cudaSuccess) return e;
  TcParams p{g.M, g.N, g.K, bn, stages, splits, num_kb, cluster_reduce ? 2 : 0, (uint32_t)ring, (int)g.epi,
             g.out_dt == DT_BF16 ? 1 : 0, g.out, g.ldo, g.bias, ws.ws, ws.counters, ws.err, (bf16*)g.vt, g.v_col0,
             g.vt_hd, g.vt_tokens, g.vt_kvp, g.vt_hkv};
  dim3 grid(tiles_n, tiles_m, splits);
  return launch_kernel(tc_gemm_kernel, grid, dim3(TC_THREADS), smem, st, cluster_reduce ? (unsigned)splits : 1u, mw,
                       mx, p);
}

}  // namespace ravel
