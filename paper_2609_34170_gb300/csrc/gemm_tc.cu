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

namespace ravel {
namespace {

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;
constexpr int TC_THREADS = 192;
constexpr uint32_t TC_A_BYTES = TC_BM * TC_BK * 2;
constexpr unsigned long long TC_TIMEOUT_NS = 1000000000ull;   // 1 s
constexpr int TC_SMEM_BUDGET = 200 * 1024;                     // operand ring
constexpr int TC_SMEM_MAX = 227 * 1024;

struct TcParams {
  int M, N, K;
  int bn, stages, splits, num_kb;
  int epi;          // Epi value, or EPI_GEGLU
  int out_bf16;
  void* out;
  int ldo;
  const float* bias;
  float* ws;
  int* counters;
  int* err;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase of `parity` to complete; false after TC_TIMEOUT_NS.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer() - t0 > TC_TIMEOUT_NS) return false;
  }
  return true;
}

__device__ __forceinline__ void tma_load_2d(const CUtensorMap* map, uint64_t* bar, void* dst, int x, int y,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(dst)),
      "l"(map), "r"(smem_u32(bar)), "r"(x), "r"(y), "l"(policy)
      : "memory");
}

// Shared-memory matrix descriptor of a K-major tile written by TMA with
// 128-byte swizzling: rows of 128 bytes, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;                 // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;       // stride byte offset: next 8-row group
  d |= (uint64_t)1 << 46;                 // descriptor version of tcgen05
  d |= (uint64_t)2 << 61;                 // 128-byte swizzle
  return d;
}

// Instruction descriptor of kind::f16 with bf16 A/B, fp32 D, both K-major.
__device__ __forceinline__ uint32_t idesc_bf16(int m, int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(acc));
}

__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float v[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Apply the epilogue to 16 consecutive tokens m0..m0+15 of weight row n.
// `xch` is the 64x16 exchange tile of the GeGLU epilogue.
__device__ __forceinline__ void apply_epilogue(const TcParams& p, int tile_n, int r, int m0, float v[16],
                                               float* xch) {
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
          if (m < p.M) o[(size_t)m * p.ldo + f] = __float2bfloat16_rn(gelu_tanh_f(v[i]) * xch[r * 17 + i]);
        }
      }
    }
    epi_bar();
    return;
  }
  const int n = tile_n * TC_BM + r;
  if (n >= p.N) return;
  const float b = p.bias ? p.bias[n] : 0.f;
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int m = m0 + i;
    if (m >= p.M) continue;
    float x = v[i] + b;
    const size_t idx = (size_t)m * p.ldo + n;
    if (p.epi == EPI_ADD_F32) {
      ((float*)p.out)[idx] += x;
    } else {
      if (p.epi == EPI_STORE_SILU) x = silu_f(x);
      if (p.out_bf16)
        ((bf16*)p.out)[idx] = __float2bfloat16_rn(x);
      else
        ((float*)p.out)[idx] = x;
    }
  }
}

__global__ void __launch_bounds__(TC_THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX, TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  const int BN = p.bn, S = p.stages;
  const uint32_t b_bytes = (uint32_t)BN * TC_BK * 2;
  uint8_t* a_s = smem;
  uint8_t* b_s = smem + (size_t)S * TC_A_BYTES;
  uint64_t* full = (uint64_t*)(b_s + (size_t)S * b_bytes);
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

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accb, 1);
    flags[0] = flags[1] = flags[2] = flags[3] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
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
      asm volatile("prefetch.tensormap [%0];" ::"l"(&tmW) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(&tmX) : "memory");
      uint64_t pol_w, pol_x;
      asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol_w));
      asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol_x));
      int i = 0;
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
  } else {
    // epilogue warps 2..5: TMEM lane quarter q = warp % 4, tile row r
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const bool ok = mbar_wait(accb, 0);
    if (!ok && lane == 0) flags[0] = 1;
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16);
    const int m_base = tile_m * BN;
    if (p.splits == 1) {
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

cudaError_t init_tc_gemm() {
  cudaError_t e = get_encoder();
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(tc_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, TC_SMEM_MAX);
}

bool tc_gemm_supported(const GemmArgs& g) {
  // TMA: 16-byte aligned bases and row strides
  if (g.K % 8 || g.lda % 8 || g.ldw % 8) return false;
  if (((uintptr_t)g.A & 15) || ((uintptr_t)g.W & 15)) return false;
  if (g.epi == EPI_GEGLU && (g.N % 128)) return false;
  return g.M > 0 && g.N > 0 && g.K > 0;
}

cudaError_t launch_gemm_tc(const GemmArgs& g, const TcWorkspace& ws, int num_sms, cudaStream_t st) {
  if (!g_encode) return cudaErrorInitializationError;
  const int bn = pick_bn(g.M);
  const int tiles_n = (g.N + TC_BM - 1) / TC_BM;
  const int tiles_m = (g.M + bn - 1) / bn;
  const int num_kb = (g.K + TC_BK - 1) / TC_BK;
  const int tiles = tiles_n * tiles_m;
  int splits = 1;
  if (tiles < num_sms) splits = std::min(num_kb, std::max(1, num_sms / tiles));
  while (splits > 1 && ((size_t)splits * tiles * bn * TC_BM * 4 > ws.ws_bytes || tiles > ws.n_counters)) --splits;
  const int stage_bytes = TC_A_BYTES + bn * TC_BK * 2;
  int stages = std::min(8, TC_SMEM_BUDGET / stage_bytes);
  stages = std::max(2, std::min(stages, std::max(2, (num_kb + splits - 1) / splits)));
  // 1024 alignment slack + operand ring + barriers / TMEM slot / flags (+ slack) + GeGLU exchange tile
  const size_t smem = 1024 + (size_t)stages * stage_bytes + (2 * stages + 1) * 8 + 128 + 64 * 17 * 4;
  CUtensorMap mw, mx;
  cudaError_t e = encode_2d(&mw, g.W, g.N, g.K, g.ldw, TC_BM);
  if (e == cudaSuccess) e = encode_2d(&mx, g.A, g.M, g.K, g.lda, bn);
  if (e != cudaSuccess) return e;
  TcParams p{g.M, g.N, g.K, bn, stages, splits, num_kb, (int)g.epi, g.out_dt == DT_BF16 ? 1 : 0, g.out, g.ldo,
             g.bias, ws.ws, ws.counters, ws.err};
  dim3 grid(tiles_n, tiles_m, splits);
  tc_gemm_kernel<<<grid, TC_THREADS, smem, st>>>(mw, mx, p);
  return cudaGetLastError();
}

}  // namespace ravel
