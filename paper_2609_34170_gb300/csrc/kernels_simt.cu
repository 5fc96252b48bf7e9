// SIMT kernels of the rolling step: weight packing, conditioning embedding,
// adaRMSNorm, action in-projection, generic projection GEMM (fp32 FFMA; the
// exact path of fp32 mode), GeGLU, grouped-query attention, and the rolling
// tail (Euler update, release, shift, Philox append).
#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "launch.h"
#include "noise.cuh"

namespace ravel {

// ============================================================================ packing

template <typename T>
__global__ void pack_transpose_kernel(const float* __restrict__ src, int K, int N, T* __restrict__ dst,
                                      int interleave64, int off) {
  __shared__ float tile[32][33];
  const int n0 = blockIdx.x * 32, k0 = blockIdx.y * 32;
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int k = k0 + i, n = n0 + threadIdx.x;
    tile[i][threadIdx.x] = (k < K && n < N) ? src[(size_t)k * N + n] : 0.f;
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int n = n0 + i, k = k0 + threadIdx.x;
    if (n < N && k < K) {
      const size_t row = interleave64 ? (size_t)(n / 64) * 128 + off + (n % 64) : (size_t)n;
      dst[row * K + k] = from_f32<T>(tile[threadIdx.x][i]);
    }
  }
}

cudaError_t launch_pack_transpose(const float* src, int K, int N, void* dst, Dtype dt, int interleave64, int off,
                                  cudaStream_t st) {
  dim3 grid((N + 31) / 32, (K + 31) / 32), block(32, 8);
  if (dt == DT_BF16)
    pack_transpose_kernel<bf16><<<grid, block, 0, st>>>(src, K, N, (bf16*)dst, interleave64, off);
  else
    pack_transpose_kernel<float><<<grid, block, 0, st>>>(src, K, N, (float*)dst, interleave64, off);
  return cudaGetLastError();
}

template <typename T>
__global__ void convert_kernel(const float* __restrict__ src, size_t n, T* __restrict__ dst) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
    dst[i] = from_f32<T>(src[i]);
}

cudaError_t launch_convert(const float* src, size_t n, void* dst, Dtype dt, cudaStream_t st) {
  const int blocks = (int)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  if (n == 0) return cudaSuccess;
  if (dt == DT_BF16)
    convert_kernel<bf16><<<blocks, 256, 0, st>>>(src, n, (bf16*)dst);
  else
    convert_kernel<float><<<blocks, 256, 0, st>>>(src, n, (float*)dst);
  return cudaGetLastError();
}

// ============================================================================ embedding

// Sinusoidal embedding of a scalar (flow time or context offset): component
// i < D/2 is sin(x w_i), i >= D/2 is cos(x w_{i-D/2}), w_i = 2 pi / p_i with
// periods p_i geometric from 4e-3 to 4 (w_i precomputed in fp64).  x w
// reaches ~1.6e3 rad, where a float32 product would already be off by ~1e-4:
// the angle is formed and reduced modulo 2 pi in fp64, then sin / cos of the
// reduced angle (|a| <= pi) in fp32.
template <typename T>
__global__ void embed_kernel(const float* __restrict__ slot_times, int H, const float* __restrict__ delta, int D,
                             const double* __restrict__ omega, T* __restrict__ E, const int* __restrict__ skip) {
  pdl_trigger();
  pdl_wait();
  if (skip && *skip) return;
  const int r = blockIdx.y;
  const double x = (r < H) ? (double)slot_times[r] : (double)delta[r - H];
  const int half = D / 2;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= half) return;
  const double ang = x * omega[i];
  const double red = ang - 6.283185307179586 * rint(ang * 0.15915494309189535);
  float s, c;
  sincosf((float)red, &s, &c);
  E[(size_t)r * D + i] = from_f32<T>(s);
  E[(size_t)r * D + half + i] = from_f32<T>(c);
}

cudaError_t launch_embed(const float* slot_times, int H, const float* delta, int B, int D, const double* omega,
                         void* E, Dtype dt, cudaStream_t st, const int* skip) {
  dim3 grid((D / 2 + 127) / 128, H + B);
  if (dt == DT_BF16)
    return launch_kernel(embed_kernel<bf16>, grid, dim3(128), 0, st, 1, slot_times, H, delta, D, omega, (bf16*)E,
                         skip);
  return launch_kernel(embed_kernel<float>, grid, dim3(128), 0, st, 1, slot_times, H, delta, D, omega, (float*)E,
                       skip);
}

// ============================================================================ conditioning cache

// One block: which rows of this step's conditioning are cached already (see
// CondCache).  The slot times hit when every one equals the cached key; a
// robot's offset hits when its value is one of the cached offsets.  Misses
// get a cache slot (a slot already referenced in this step is never taken;
// with no slot left the robot keeps this step's fresh row), and their keys
// are written now: the rows themselves arrive through cond_commit before
// any reader of this step, and a later step reads them only after that.
__global__ void cond_check_kernel(CondArgs a) {
  __shared__ int s_tmiss;
  __shared__ unsigned s_ref;   // cache slots referenced by this step
  pdl_trigger();
  pdl_wait();
  CondCache* cc = a.cc;
  if (threadIdx.x == 0) {
    s_tmiss = a.enabled ? !cc->t_valid : 1;
    s_ref = 0u;
  }
  __syncthreads();
  for (int j = threadIdx.x; j < a.H; j += blockDim.x)
    if (a.slot_times[j] != a.t_key[j]) s_tmiss = 1;   // benign race: every writer stores 1
  // offsets: look up in parallel; -1 = miss
  for (int b = threadIdx.x; b < a.B; b += blockDim.x) {
    int row = -1;
    if (a.enabled) {
      const float d = a.delta[b];
      for (int c = 0; c < kCondCache; ++c)
        if (cc->used[c] && cc->delta[c] == d) {
          row = a.H + a.Bmax + c;
          atomicOr(&s_ref, 1u << c);
          break;
        }
    }
    a.drow[b] = row;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int any_miss = s_tmiss, nc = 0;
    unsigned ref = s_ref;
    for (int b = 0; b < a.B; ++b) {
      if (a.drow[b] >= 0) continue;
      any_miss = 1;
      const float d = a.delta[b];
      int row = a.H + b;   // this step's fresh row unless a cache slot is found
      if (a.enabled) {
        int c = -1;
        for (int k = 0; k < kCondCache; ++k)   // assigned to an earlier robot of this step?
          if ((ref >> k & 1u) && cc->used[k] && cc->delta[k] == d) c = k;
        if (c < 0) {
          for (int k = 0; k < kCondCache && c < 0; ++k) {
            const int v = (cc->next + k) % kCondCache;
            if (!(ref >> v & 1u)) c = v;
          }
          if (c >= 0) {
            cc->next = (c + 1) % kCondCache;
            cc->delta[c] = d;
            cc->used[c] = 1;
            a.commit[2 * nc] = a.H + b;
            a.commit[2 * nc + 1] = a.H + a.Bmax + c;
            ++nc;
          }
        }
        if (c >= 0) {
          ref |= 1u << c;
          row = a.H + a.Bmax + c;
        }
      }
      a.drow[b] = row;
    }
    cc->n_commit = nc;
    cc->skip = any_miss ? 0 : 1;
    if (a.enabled) cc->t_valid = 1;
  }
  // the slot times become the key (a miss recomputes rows [0, H) this step)
  if (a.enabled)
    for (int j = threadIdx.x; j < a.H; j += blockDim.x) a.t_key[j] = a.slot_times[j];
}

cudaError_t launch_cond_check(const CondArgs& a, cudaStream_t st) {
  return launch_kernel(cond_check_kernel, dim3(1), dim3(256), 0, st, 1, a);
}

// Copies the rows that cond_check listed (this step's fresh offset rows) into
// their cache slots.
__global__ void cond_commit_kernel(CondArgs a) {
  pdl_trigger();
  pdl_wait();
  const int n = a.cc->n_commit;
  for (int i = 0; i < n; ++i) {
    const float4* src = (const float4*)(a.modv + (size_t)a.commit[2 * i] * a.mod_ld);
    float4* dst = (float4*)(a.modv + (size_t)a.commit[2 * i + 1] * a.mod_ld);
    for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < a.mod_ld / 4; c += gridDim.x * blockDim.x) dst[c] = src[c];
  }
}

cudaError_t launch_cond_commit(const CondArgs& a, cudaStream_t st) {
  return launch_kernel(cond_commit_kernel, dim3(64), dim3(256), 0, st, 1, a);
}

// ============================================================================ GEMM (SIMT)

// 64x64 output tile, K step 32, 256 threads, 4x4 outputs per thread spread
// with stride 16 so that shared-memory reads are broadcast-friendly.
template <typename T, int EPI, typename TO>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ A, int lda, const T* __restrict__ W,
                                                        int ldw, int M, int N, int K, TO* __restrict__ out, int ldo,
                                                        const float* __restrict__ bias, const int* __restrict__ skip) {
  pdl_trigger();
  pdl_wait();
  if (skip && *skip) return;
  __shared__ float As[32][64 + 4];
  __shared__ float Ws[32][64 + 4];
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 32) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int idx = threadIdx.x + 256 * i;
      const int r = idx >> 5, kk = idx & 31;
      const int m = m0 + r, n = n0 + r, k = k0 + kk;
      As[kk][r] = (m < M && k < K) ? to_f32(A[(size_t)m * lda + k]) : 0.f;
      Ws[kk][r] = (n < N && k < K) ? to_f32(W[(size_t)n * ldw + k]) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < 32; ++kk) {
      float a[4], w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < 4; ++j) w[j] = Ws[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], w[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty + 16 * i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx + 16 * j;
      if (n >= N) continue;
      float v = acc[i][j] + (bias ? bias[n] : 0.f);
      if (EPI == EPI_STORE_SILU) v = silu_f(v);
      if (EPI == EPI_ADD_F32)
        ((float*)out)[(size_t)m * ldo + n] += v;
      else
        out[(size_t)m * ldo + n] = from_f32<TO>(v);
    }
  }
}

template <typename T>
static cudaError_t gemm_simt_dispatch(const GemmArgs& g, cudaStream_t st) {
  dim3 grid((g.N + 63) / 64, (g.M + 63) / 64);
  const T* A = (const T*)g.A;
  const T* W = (const T*)g.W;
  if (g.epi == EPI_ADD_F32) {
    launch_kernel(gemm_simt_kernel<T, EPI_ADD_F32, float>, grid, dim3(256), 0, st, 1, A, g.lda, W, g.ldw, g.M, g.N, g.K, (float*)g.out,
                                                                 g.ldo, g.bias, g.skip);
  } else if (g.out_dt == DT_BF16) {
    if (g.epi == EPI_STORE_SILU)
      launch_kernel(gemm_simt_kernel<T, EPI_STORE_SILU, bf16>, grid, dim3(256), 0, st, 1, A, g.lda, W, g.ldw, g.M, g.N, g.K,
                                                                     (bf16*)g.out, g.ldo, g.bias, g.skip);
    else
      launch_kernel(gemm_simt_kernel<T, EPI_STORE, bf16>, grid, dim3(256), 0, st, 1, A, g.lda, W, g.ldw, g.M, g.N, g.K, (bf16*)g.out,
                                                                g.ldo, g.bias, g.skip);
  } else {
    if (g.epi == EPI_STORE_SILU)
      launch_kernel(gemm_simt_kernel<T, EPI_STORE_SILU, float>, grid, dim3(256), 0, st, 1, A, g.lda, W, g.ldw, g.M, g.N, g.K,
                                                                      (float*)g.out, g.ldo, g.bias, g.skip);
    else
      launch_kernel(gemm_simt_kernel<T, EPI_STORE, float>, grid, dim3(256), 0, st, 1, A, g.lda, W, g.ldw, g.M, g.N, g.K, (float*)g.out,
                                                                 g.ldo, g.bias, g.skip);
  }
  return cudaGetLastError();
}

cudaError_t launch_gemm_simt(const GemmArgs& g, Dtype dt, cudaStream_t st) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  return dt == DT_BF16 ? gemm_simt_dispatch<bf16>(g, st) : gemm_simt_dispatch<float>(g, st);
}

// ============================================================================ adaRMSNorm

__device__ __forceinline__ float4 ld4(const float* p) { return *(const float4*)p; }
__device__ __forceinline__ float4 add3(float4 a, float4 b, float4 c) {
  return make_float4(a.x + b.x + c.x, a.y + b.y + c.y, a.z + b.z + c.z, a.w + b.w + c.w);
}
__device__ __forceinline__ void st4(float* p, float4 v) { *(float4*)p = v; }
__device__ __forceinline__ void st4(bf16* p, float4 v) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
  uint2 u;
  u.x = *(uint32_t*)&lo;
  u.y = *(uint32_t*)&hi;
  *(uint2*)p = u;
}

__device__ __forceinline__ float4 add2(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float4 ld4(const bf16* p) {
  const uint2 u = *(const uint2*)p;
  const __nv_bfloat162 lo = *(const __nv_bfloat162*)&u.x, hi = *(const __nv_bfloat162*)&u.y;
  return make_float4(__low2float(lo), __high2float(lo), __low2float(hi), __high2float(hi));
}

// adaRMSNorm over a block of rows of one robot (Sec. 3.1, Eq. 2):
//   action row (b, j):  y = x * rsqrt(mean(x^2) + eps) * (1 + scale) + shift,
//                       (scale, shift) = M_t[j] + M_delta[b] + bias  (the
//                       modulation is linear in the two embeddings)
//   FOP row (b, f):     y = z * rsqrt(mean(z^2) + eps) * (1 + gamma)
// A thread owns columns 4*tid + 1024*g (g < G) of every row of the block, so
// the per-robot part M_delta[b] + bias (or gamma) is read once per block and
// kept in registers; rows go through one at a time with one barrier each
// (the row sums are reduced through a double-buffered table).  Few rows per
// block: the row's loads are the block's critical path, and spreading the
// rows over more blocks (one each when they fit the SMs) beat batching four
// rows per round trip.
template <typename T, int G>
__global__ void __launch_bounds__(256) ada_norm_kernel(NormArgs a, int rb_act, int nb_act, int rb_fop, int nb_fop) {
  constexpr int R = 1;
  __shared__ float red[2][R][8];
  pdl_trigger();
  const int D = a.D, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int blk = blockIdx.x;
  const bool act = blk < a.B * nb_act;
  int b, j0, j1;
  if (act) {
    b = blk / nb_act;
    j0 = (blk % nb_act) * rb_act;
    j1 = min(a.H, j0 + rb_act);
  } else {
    blk -= a.B * nb_act;
    b = blk / nb_fop;
    j0 = (blk % nb_fop) * rb_fop;
    j1 = min(a.F, j0 + rb_fop);
  }
  float4 csc[G], csh[G];   // action: bias (+ M_delta[b] after the wait); FOP: gamma
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const int c = 4 * threadIdx.x + 1024 * g;
    csc[g] = csh[g] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (c < D) {   // weights: independent of the earlier kernels
      if (act && !a.act_gain) {
        csc[g] = ld4(a.mod_b + a.off + c);
        csh[g] = ld4(a.mod_b + a.off + D + c);
      } else {
        csc[g] = ld4(act ? a.act_gain + c : a.gamma + c);
      }
    }
  }
  pdl_wait();
  const bool modulated = act && !a.act_gain;   // action rows with adaLN modulation
  const float* md = modulated ? a.modv + (size_t)(a.drow ? a.drow[b] : a.H + b) * a.mod_ld + a.off : nullptr;
  int buf = 0;
  for (int j = j0; j < j1; j += R, buf ^= 1) {
    float4 xv[R][G], ts[R][G], th[R][G];
    float ss[R];
    if (modulated && j == j0) {   // M_delta[b] joins the first batch's loads (one round trip)
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const int c = 4 * threadIdx.x + 1024 * g;
        if (c < D) {
          csc[g] = add2(csc[g], ld4(md + c));
          csh[g] = add2(csh[g], ld4(md + D + c));
        }
      }
    }
#pragma unroll
    for (int rr = 0; rr < R; ++rr) {
      ss[rr] = 0.f;
      const int jj = j + rr;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const int c = 4 * threadIdx.x + 1024 * g;
        xv[rr][g] = ts[rr][g] = th[rr][g] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (jj < j1 && c < D) {
          if (act) {
            xv[rr][g] = ld4(a.x + (size_t)(b * a.H + jj) * D + c);
            if (modulated) {
              const float* mt = a.modv + (size_t)(b * a.t_stride + jj) * a.mod_ld + a.off;
              ts[rr][g] = ld4(mt + c);
              th[rr][g] = ld4(mt + D + c);
            }
          } else {
            xv[rr][g] = ld4((const T*)a.fop + (size_t)(b * a.F + jj) * D + c);
          }
        }
      }
#pragma unroll
      for (int g = 0; g < G; ++g)
        ss[rr] += xv[rr][g].x * xv[rr][g].x + xv[rr][g].y * xv[rr][g].y + xv[rr][g].z * xv[rr][g].z +
                  xv[rr][g].w * xv[rr][g].w;
    }
#pragma unroll
    for (int rr = 0; rr < R; ++rr) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ss[rr] += __shfl_xor_sync(0xffffffffu, ss[rr], o);
      if (lane == 0) red[buf][rr][warp] = ss[rr];
    }
    __syncthreads();
#pragma unroll
    for (int rr = 0; rr < R; ++rr) {
      const int jj = j + rr;
      float tot = 0.f;
#pragma unroll
      for (int w = 0; w < 8; ++w) tot += red[buf][rr][w];
      const float inv = rsqrtf(tot / (float)D + 1e-6f);
      if (jj >= j1) continue;
      T* Y = (T*)a.Y + ((size_t)b * a.row_pitch + (act ? jj : a.H + jj)) * D;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const int c = 4 * threadIdx.x + 1024 * g;
        if (c >= D) continue;
        const float4 x = xv[rr][g];
        if (modulated) {
          const float4 sc = add2(csc[g], ts[rr][g]), sh = add2(csh[g], th[rr][g]);
          st4(Y + c, make_float4(x.x * inv * (1.f + sc.x) + sh.x, x.y * inv * (1.f + sc.y) + sh.y,
                                 x.z * inv * (1.f + sc.z) + sh.z, x.w * inv * (1.f + sc.w) + sh.w));
        } else {
          const float4 gm = csc[g];
          st4(Y + c, make_float4(x.x * inv * (1.f + gm.x), x.y * inv * (1.f + gm.y), x.z * inv * (1.f + gm.z),
                                 x.w * inv * (1.f + gm.w)));
        }
      }
    }
  }
}

namespace {
int g_norm_sms = 0;
}

template <typename T>
cudaError_t launch_ada_norm_t(const NormArgs& a, cudaStream_t st) {
  if (!g_norm_sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&g_norm_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || g_norm_sms < 1)
      g_norm_sms = 132;
  }
  const int G = (a.D + 1023) / 1024;
  const int R = 1;
  // rows per block: as few as fill up to 8 resident blocks of 256 threads per
  // SM (one row each when the rows fit)
  const int nf = a.fop ? a.F : 0;
  const int total = a.B * (a.H + nf);
  int rb_all = (total + 8 * g_norm_sms - 1) / (8 * g_norm_sms);
  rb_all = (rb_all + R - 1) / R * R;
  auto rows_per_block = [&](int rows_per_robot) { return std::max(R, std::min(rb_all, rows_per_robot)); };
  const int rb_act = rows_per_block(a.H), nb_act = (a.H + rb_act - 1) / rb_act;
  const int rb_fop = nf ? rows_per_block(nf) : 1, nb_fop = nf ? (nf + rb_fop - 1) / rb_fop : 0;
  const int blocks = a.B * (nb_act + nb_fop);
  if (blocks <= 0) return cudaSuccess;
  NormArgs b = a;
  b.F = nf;
  switch (G) {
    case 1: return launch_kernel(ada_norm_kernel<T, 1>, dim3(blocks), dim3(256), 0, st, 1, b, rb_act, nb_act, rb_fop, nb_fop);
    case 2: return launch_kernel(ada_norm_kernel<T, 2>, dim3(blocks), dim3(256), 0, st, 1, b, rb_act, nb_act, rb_fop, nb_fop);
    case 3: return launch_kernel(ada_norm_kernel<T, 3>, dim3(blocks), dim3(256), 0, st, 1, b, rb_act, nb_act, rb_fop, nb_fop);
    default: return launch_kernel(ada_norm_kernel<T, 4>, dim3(blocks), dim3(256), 0, st, 1, b, rb_act, nb_act, rb_fop, nb_fop);
  }
}

cudaError_t launch_ada_norm(const NormArgs& a, Dtype dt, cudaStream_t st) {
  if (a.D <= 0 || a.D > 4096 || a.D % 4) return cudaErrorInvalidValue;
  return dt == DT_BF16 ? launch_ada_norm_t<bf16>(a, st) : launch_ada_norm_t<float>(a, st);
}

// ============================================================================ in-proj

__global__ void in_proj_kernel(const float* __restrict__ buf, int A, int D, const float* __restrict__ in_w,
                               const float* __restrict__ in_b, float* __restrict__ x, const float* __restrict__ state,
                               const float* __restrict__ rel_mask, const float* __restrict__ slot_times, int H,
                               int t_stride) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float arow[];   // the action row of this slot
  const int r = blockIdx.y;
  for (int i = threadIdx.x; i < A; i += blockDim.x) {
    float a = buf[(size_t)r * A + i];
    if (state) {   // relative coordinates of the expert: a - (1 - t_j) m s_b
      const int b = r / H, j = r % H;
      a = __fsub_rn(a, __fmul_rn(__fsub_rn(1.f, slot_times[b * t_stride + j]),
                                 __fmul_rn(rel_mask[i], state[(size_t)b * A + i])));
    }
    arow[i] = a;
  }
  __syncthreads();
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= D) return;
  float acc = in_b[c];
  for (int i = 0; i < A; ++i) acc = fmaf(arow[i], in_w[(size_t)i * D + c], acc);
  x[(size_t)r * D + c] = acc;
}

cudaError_t launch_in_proj(const float* buf, int BH, int A, int D, const float* in_w, const float* in_b, float* x,
                           cudaStream_t st, const float* state, const float* rel_mask, const float* slot_times, int H,
                           int t_stride) {
  if (BH <= 0) return cudaSuccess;
  return launch_kernel(in_proj_kernel, dim3((D + 255) / 256, BH), dim3(256), A * sizeof(float), st, 1, buf, A, D,
                       in_w, in_b, x, state, rel_mask, slot_times, H, t_stride);
}

// The in-projection of whole rows with the first layer's adaRMSNorm: one
// CTA per row; an action row is projected (x, fp32), then normalised with its
// modulation into Y; a FOP row is normalised with its gain.  (Rows of up to
// 4096 features: a thread owns features tid, tid + 256, ...)
template <typename T>
__global__ void __launch_bounds__(256) in_proj_norm_kernel(const float* __restrict__ buf, int A, int D,
                                                           const float* __restrict__ in_w,
                                                           const float* __restrict__ in_b, float* __restrict__ x,
                                                           const float* __restrict__ state,
                                                           const float* __restrict__ rel_mask,
                                                           const float* __restrict__ slot_times, RowNorm rn) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float arow[];   // the action row of this slot
  __shared__ float red[32];
  const int r = blockIdx.x, BH = rn.B * rn.H;
  float v[16];
  float ss = 0.f;
  if (r < BH) {
    const int b = r / rn.H, j = r % rn.H;
    for (int i = threadIdx.x; i < A; i += blockDim.x) {
      float a = buf[(size_t)r * A + i];
      if (state)   // relative coordinates of the expert: a - (1 - t_j) m s_b
        a = __fsub_rn(a, __fmul_rn(__fsub_rn(1.f, slot_times[b * rn.t_stride + j]),
                                   __fmul_rn(rel_mask[i], state[(size_t)b * A + i])));
      arow[i] = a;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const int c = threadIdx.x + 256 * k;
      v[k] = 0.f;
      if (c < D) {
        float acc = in_b[c];
        for (int i = 0; i < A; ++i) acc = fmaf(arow[i], in_w[(size_t)i * D + c], acc);
        x[(size_t)r * D + c] = acc;
        v[k] = acc;
        ss += acc * acc;
      }
    }
    const float inv = rsqrtf(block_sum(ss, red) / (float)D + 1e-6f);
    const float* mt = rn.modv + (size_t)(b * rn.t_stride + j) * rn.mod_ld + rn.off;
    const float* md = rn.modv + (size_t)(rn.drow ? rn.drow[b] : rn.H + b) * rn.mod_ld + rn.off;
    const float* mb = rn.mod_b + rn.off;
    T* Y = (T*)rn.Y + (size_t)(b * rn.row_pitch + j) * D;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const int c = threadIdx.x + 256 * k;
      if (c < D) {
        const float sc = mt[c] + md[c] + mb[c], sh = mt[D + c] + md[D + c] + mb[D + c];
        Y[c] = from_f32<T>(v[k] * inv * (1.f + sc) + sh);
      }
    }
  } else {
    const int fr = r - BH, b = fr / rn.F, f = fr % rn.F;
    const T* z = (const T*)rn.fop + (size_t)(b * rn.F + f) * D;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const int c = threadIdx.x + 256 * k;
      v[k] = c < D ? to_f32(z[c]) : 0.f;
      ss += v[k] * v[k];
    }
    const float inv = rsqrtf(block_sum(ss, red) / (float)D + 1e-6f);
    T* Y = (T*)rn.Y + (size_t)(b * rn.row_pitch + rn.H + f) * D;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const int c = threadIdx.x + 256 * k;
      if (c < D) Y[c] = from_f32<T>(v[k] * inv * (1.f + rn.gamma[c]));
    }
  }
}

cudaError_t launch_in_proj_norm(const float* buf, int A, int D, const float* in_w, const float* in_b, float* x,
                                const float* state, const float* rel_mask, const float* slot_times, const RowNorm& rn,
                                Dtype dt, cudaStream_t st) {
  if (D > 4096) return cudaErrorInvalidValue;
  const int rows = rn.B * rn.H + (rn.fop ? rn.B * rn.F : 0);
  if (rows <= 0) return cudaSuccess;
  if (dt == DT_BF16)
    return launch_kernel(in_proj_norm_kernel<bf16>, dim3(rows), dim3(256), A * sizeof(float), st, 1, buf, A, D, in_w,
                         in_b, x, state, rel_mask, slot_times, rn);
  return launch_kernel(in_proj_norm_kernel<float>, dim3(rows), dim3(256), A * sizeof(float), st, 1, buf, A, D, in_w,
                       in_b, x, state, rel_mask, slot_times, rn);
}

__global__ void noop_kernel() {}

cudaError_t launch_noop(cudaStream_t st) { return launch_kernel(noop_kernel, dim3(1), dim3(1), 0, st, 1); }

// ============================================================================ GeGLU

template <typename T>
__global__ void geglu_kernel(const float* __restrict__ GU, int M, int Fm, T* __restrict__ Hm) {
  pdl_trigger();
  pdl_wait();
  const size_t total = (size_t)M * Fm;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total; i += (size_t)gridDim.x * blockDim.x) {
    const int m = (int)(i / Fm), f = (int)(i % Fm);
    const size_t base = (size_t)m * 2 * Fm + (size_t)(f / 64) * 128 + (f % 64);
    Hm[i] = from_f32<T>(gelu_tanh_f(GU[base]) * GU[base + 64]);
  }
}

cudaError_t launch_geglu(const float* GU, int M, int Fm, void* Hm, Dtype dt, cudaStream_t st) {
  const size_t total = (size_t)M * Fm;
  if (!total) return cudaSuccess;
  const int blocks = (int)((total + 255) / 256 < 8192 ? (total + 255) / 256 : 8192);
  if (dt == DT_BF16) return launch_kernel(geglu_kernel<bf16>, dim3(blocks), dim3(256), 0, st, 1, GU, M, Fm, (bf16*)Hm);
  return launch_kernel(geglu_kernel<float>, dim3(blocks), dim3(256), 0, st, 1, GU, M, Fm, (float*)Hm);
}

// ============================================================================ attention (SIMT)

// One CTA per (robot b, KV head g, tile of QT query rows).  Query row r of a
// (b, g) pair is slot j = r / G of query head g*G + r % G.  Keys are visited
// in chunks of KT: [0, P) the active context's prefix, [P, P+F) the FOP
// tokens, [P+F, P+F+H) the action slots; online softmax in fp32.
constexpr int ATT_QT = 16, ATT_KT = 32, ATT_THREADS = 256;

template <typename T>
__global__ void __launch_bounds__(ATT_THREADS) attention_simt_kernel(AttnArgs a) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float sm[];
  const int hd = a.hd;
  float* Qs = sm;                      // [QT][hd]
  float* Ks = Qs + ATT_QT * hd;        // [KT][hd]
  float* Vs = Ks + ATT_KT * hd;        // [KT][hd]
  float* Ss = Vs + ATT_KT * hd;        // [QT][KT]
  const int bg = blockIdx.x;
  const int b = bg / a.Hkv, g = bg % a.Hkv;
  const int G = a.Hq / a.Hkv;
  const int nrows = a.H * G;
  const int r0 = blockIdx.y * ATT_QT;
  const int slot = a.ctx_state[2 * b];       // this robot's active context
  const int P = a.ctx_state[2 * b + 1];
  if (P < 0 || P > a.Pmax) {
    if (threadIdx.x == 0) raise_error(a.err, ERR_PREFIX_LEN);
    return;
  }
  const T* qkv = (const T*)a.qkv;
  const size_t ctx_off = ((((size_t)a.layer * a.Bmax + b) * a.Hkv + g) * (size_t)a.Pmax) * hd;
  const T* pk = (const T*)(slot ? a.ctx_k1 : a.ctx_k0) + ctx_off;
  const T* pv = (const T*)(slot ? a.ctx_v1 : a.ctx_v0) + ctx_off;
  const int kofs = a.Hq * hd + g * hd, vofs = (a.Hq + a.Hkv) * hd + g * hd;
  const int nk = P + a.F + a.H;
  const int rpr = a.H + a.F;   // QKV rows per robot: H action slots, then F FOP tokens
  const float scale = rsqrtf((float)hd);

  for (int i = threadIdx.x; i < ATT_QT * hd; i += ATT_THREADS) {
    const int rr = i / hd, c = i % hd, r = r0 + rr;
    float v = 0.f;
    if (r < nrows) {
      const int j = r / G, h = g * G + r % G;
      v = to_f32(qkv[(size_t)(b * rpr + j) * a.ld_qkv + h * hd + c]);
    }
    Qs[i] = v * scale;
  }
  // thread layout for scores / softmax: 16 threads per query row
  const int srow = threadIdx.x >> 4, slane = threadIdx.x & 15;
  float m_run = -INFINITY, l_run = 0.f;
  // output accumulators: row orow, columns ocol + 16*i
  const int orow = threadIdx.x >> 4, ocol = threadIdx.x & 15;
  float acc[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) acc[i] = 0.f;
  const int qrow_slot = (r0 + srow < nrows) ? (r0 + srow) / G : -1;

  for (int k0 = 0; k0 < nk; k0 += ATT_KT) {
    __syncthreads();
    for (int i = threadIdx.x; i < ATT_KT * hd; i += ATT_THREADS) {
      const int kk = i / hd, c = i % hd, key = k0 + kk;
      float kv = 0.f, vv = 0.f;
      if (key < P) {
        kv = to_f32(pk[(size_t)key * hd + c]);
        vv = to_f32(pv[(size_t)key * hd + c]);
      } else if (key < P + a.F) {
        const size_t row = (size_t)(b * rpr + a.H + (key - P)) * a.ld_qkv;
        kv = to_f32(qkv[row + kofs + c]);
        vv = to_f32(qkv[row + vofs + c]);
      } else if (key < nk) {
        const size_t row = (size_t)(b * rpr + (key - P - a.F)) * a.ld_qkv;
        kv = to_f32(qkv[row + kofs + c]);
        vv = to_f32(qkv[row + vofs + c]);
      }
      Ks[i] = kv;
      Vs[i] = vv;
    }
    __syncthreads();
    // scores: row srow, keys slane and slane + 16
    float s[2];
#pragma unroll
    for (int t = 0; t < 2; ++t) {
      const int kk = slane + 16 * t, key = k0 + kk;
      float d = 0.f;
      for (int c = 0; c < hd; ++c) d = fmaf(Qs[srow * hd + c], Ks[kk * hd + c], d);
      bool vis = key < nk;
      if (a.mask_mode == 1 && key >= P + a.F && key < nk) vis = vis && (key - P - a.F == qrow_slot);
      s[t] = vis ? d : -INFINITY;
    }
    float cmax = fmaxf(s[0], s[1]);
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) cmax = fmaxf(cmax, __shfl_xor_sync(0xffffffffu, cmax, o));
    const float m_new = fmaxf(m_run, cmax);
    const float corr = (m_new == -INFINITY) ? 1.f : __expf(m_run - m_new);
    float psum = 0.f;
#pragma unroll
    for (int t = 0; t < 2; ++t) {
      const float p = (s[t] == -INFINITY) ? 0.f : __expf(s[t] - m_new);
      Ss[srow * ATT_KT + slane + 16 * t] = p;
      psum += p;
    }
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, o);
    l_run = l_run * corr + psum;
    m_run = m_new;
    __syncthreads();
    // P V: orow == srow, so corr is this thread's own row correction
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int c = ocol + 16 * i;
      if (c < hd) {
        float v = acc[i] * corr;
        for (int kk = 0; kk < ATT_KT; ++kk) v = fmaf(Ss[orow * ATT_KT + kk], Vs[kk * hd + c], v);
        acc[i] = v;
      }
    }
  }
  const int r = r0 + orow;
  if (r < nrows) {
    const int j = r / G, h = g * G + r % G;
    T* o = (T*)a.out + (size_t)(b * a.H + j) * a.ld_out + h * hd;
    const float inv = 1.f / l_run;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int c = ocol + 16 * i;
      if (c < hd) o[c] = from_f32<T>(acc[i] * inv);
    }
  }
}

cudaError_t launch_attention_simt(const AttnArgs& a, Dtype dt, cudaStream_t st) {
  if (a.hd > 256 || a.hd % 8) return cudaErrorInvalidValue;
  const int G = a.Hq / a.Hkv;
  dim3 grid(a.B * a.Hkv, (a.H * G + ATT_QT - 1) / ATT_QT);
  const size_t smem = (size_t)(ATT_QT * a.hd + 2 * ATT_KT * a.hd + ATT_QT * ATT_KT) * sizeof(float);
  if (dt == DT_BF16) return launch_kernel(attention_simt_kernel<bf16>, grid, dim3(ATT_THREADS), smem, st, 1, a);
  return launch_kernel(attention_simt_kernel<float>, grid, dim3(ATT_THREADS), smem, st, 1, a);
  return cudaGetLastError();
}

// ============================================================================ FOP adapter cross-attention

// One CTA per (robot b, query head h); warp w takes slots w, w + 8, ...: the
// scores of a slot over the F FOP keys (lanes split the head dim), the
// softmax, and the lanes' head-dim slices of the weighted values.
template <typename T>
__global__ void __launch_bounds__(256) fop_xattn_kernel(const T* __restrict__ Q, const T* __restrict__ KV,
                                                        T* __restrict__ out, int H, int F, int Hq, int Hkv, int hd,
                                                        const float* __restrict__ gate) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float xs[];
  float* Ks = xs;                 // [F][hd]
  float* Vs = Ks + F * hd;        // [F][hd]
  float* Ps = Vs + F * hd;        // [8 warps][F]
  const int b = blockIdx.x / Hq, h = blockIdx.x % Hq, g = h / (Hq / Hkv);
  const int ldkv = 2 * Hkv * hd, ldq = Hq * hd;
  for (int i = threadIdx.x; i < F * hd; i += blockDim.x) {
    const int f = i / hd, c = i % hd;
    const T* row = KV + (size_t)(b * F + f) * ldkv;
    Ks[i] = to_f32(row[g * hd + c]);
    Vs[i] = to_f32(row[Hkv * hd + g * hd + c]);
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float scale = rsqrtf((float)hd), gt = tanhf(gate[0]);
  float* p = Ps + warp * F;
  for (int j = warp; j < H; j += 8) {
    const T* q = Q + (size_t)(b * H + j) * ldq + h * hd;
    float mx = -INFINITY;
    for (int f = 0; f < F; ++f) {
      float d = 0.f;
      for (int c = lane; c < hd; c += 32) d = fmaf(to_f32(q[c]), Ks[f * hd + c], d);
      d = warp_sum(d) * scale;
      if (lane == 0) p[f] = d;
      mx = fmaxf(mx, d);
    }
    __syncwarp();
    float sum = 0.f;
    for (int f = 0; f < F; ++f) sum += __expf(p[f] - mx);
    const float inv = gt / sum;
    T* o = out + (size_t)(b * H + j) * ldq + h * hd;
    for (int c = lane; c < hd; c += 32) {
      float acc = 0.f;
      for (int f = 0; f < F; ++f) acc = fmaf(__expf(p[f] - mx), Vs[f * hd + c], acc);
      o[c] = from_f32<T>(acc * inv);
    }
    __syncwarp();
  }
}

cudaError_t launch_fop_xattn(const void* Q, const void* KV, void* out, int B, int H, int F, int Hq, int Hkv, int hd,
                             const float* gate, Dtype dt, cudaStream_t st) {
  if (B <= 0 || H <= 0) return cudaSuccess;
  if (F < 1 || F > 64 || hd > 256) return cudaErrorInvalidValue;
  const size_t smem = ((size_t)2 * F * hd + 8 * F) * sizeof(float);
  if (dt == DT_BF16)
    return launch_kernel(fop_xattn_kernel<bf16>, dim3(B * Hq), dim3(256), smem, st, 1, (const bf16*)Q,
                         (const bf16*)KV, (bf16*)out, H, F, Hq, Hkv, hd, gate);
  return launch_kernel(fop_xattn_kernel<float>, dim3(B * Hq), dim3(256), smem, st, 1, (const float*)Q,
                       (const float*)KV, (float*)out, H, F, Hq, Hkv, hd, gate);
}

// ============================================================================ tail

// One CTA per robot: a'_j = a_j + dt_j v_j (Eq. 3), released = a'_0, buffer
// slots shift forward, the last slot receives the Gaussian action of index
// counters[b], and the counter advances.
// Euler step, release, shift and noise append of robot b (Eq. 3 and the roll
// after it), by the whole block; sa: H*A floats of shared memory.
__device__ void tail_robot(const TailArgs& a, int b, float* sa) {
  const int H = a.H, A = a.A;
  float* buf = a.buffer + (size_t)b * H * A;
  const float* v = a.vel + (size_t)b * H * A;
  for (int i = threadIdx.x; i < H * A; i += blockDim.x) {
    const int j = i / A;
    const float* tb = a.slot_times + (size_t)b * a.t_stride;   // robot b's schedule
    const float t1 = tb[j];
    const float t0 = j ? tb[j - 1] : 0.f;
    const float dt = __fsub_rn(t1, t0);
    // absolute buffer, relative expert: the slot also moves by dt m s as its
    // flow time drops from t_j to t_{j-1}
    const float vi = __ldcg(v + i);   // (written by other CTAs of the fused head kernel)
    const float vv = a.state ? fmaf(a.rel_mask[i % A], a.state[(size_t)b * A + i % A], vi) : vi;
    sa[i] = fmaf(dt, vv, buf[i]);
    if (a.vel_out) a.vel_out[(size_t)b * H * A + i] = vi;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < H * A; i += blockDim.x) {
    if (i < A) a.released[(size_t)b * A + i] = sa[i];
    if (i < (H - 1) * A) buf[i] = sa[i + A];
  }
  const uint64_t n = a.counters[b];
  const uint64_t seed = a.seeds[b];
  for (int g = threadIdx.x; g < (A + 3) / 4; g += blockDim.x) {
    float z[4];
    action_noise4(seed, n, (uint32_t)g, z);
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (4 * g + i < A) buf[(size_t)(H - 1) * A + 4 * g + i] = z[i];
  }
  __syncthreads();
  if (threadIdx.x == 0) a.counters[b] = n + 1;
}

__global__ void tail_kernel(TailArgs a) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float sa[];   // [H][A]
  tail_robot(a, blockIdx.x, sa);
}

cudaError_t launch_tail(const TailArgs& a, cudaStream_t st) {
  if (a.B <= 0) return cudaSuccess;
  const size_t smem = (size_t)a.H * a.A * sizeof(float);
  return launch_kernel(tail_kernel, dim3(a.B), dim3(256), smem, st, 1, a);
}

// The step's last three stages in one launch (bf16 mode, A <= 32): the final
// adaRMSNorm of each action row (Eq. 2's modulation, offset fin_off), the
// velocity head v = Y W_out^T + b_out on the bf16-rounded normed row (as the
// separate norm + GEMM compute it), and, by the CTA of each robot that
// finishes last, the Euler step, release, shift and noise append (tail_robot).
// A CTA owns rows_per_cta slots of one robot; the robot's CTAs count their
// finished rows on cnt[b] (reset by the last one, so it is zero between
// launches), the classic last-block pattern: no CTA waits for another.
template <bool FULL>   // FULL: A == 32
__global__ void __launch_bounds__(256) head_tail_kernel(HeadArgs h, TailArgs a) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[8][33];     // per-warp sums: [warp][output] (+ the norm's row sum in [w][32])
  __shared__ int last;
  extern __shared__ float sa[];    // [H][A], the last CTA's tail
  const int nb = (a.H + h.rows_per_cta - 1) / h.rows_per_cta;
  const int b = blockIdx.x / nb, j0 = (blockIdx.x % nb) * h.rows_per_cta;
  const int j1 = min(a.H, j0 + h.rows_per_cta);
  const int D = h.D, A = a.A, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* md = h.modv + (size_t)(h.drow ? h.drow[b] : a.H + b) * h.mod_ld + h.off;
  const float* mb = h.mod_b + h.off;
  for (int j = j0; j < j1; ++j) {
    const float* xr = h.x + (size_t)(b * a.H + j) * D;
    const float* mt = h.modv + (size_t)(b * h.t_stride + j) * h.mod_ld + h.off;
    // sum of squares of the row (4 features per thread per pass)
    float ss = 0.f;
    for (int f = 4 * threadIdx.x; f < D; f += 4 * blockDim.x) {
      const float4 xv = *(const float4*)(xr + f);
      ss += xv.x * xv.x + xv.y * xv.y + xv.z * xv.z + xv.w * xv.w;
    }
    ss = warp_sum(ss);
    if (lane == 0) red[warp][32] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += red[w][32];
    const float inv = rsqrtf(tot / (float)D + 1e-6f);
    // this thread's partial products for all 32 outputs
    float acc[32];
#pragma unroll
    for (int o = 0; o < 32; ++o) acc[o] = 0.f;
    for (int f = 4 * threadIdx.x; f < D; f += 4 * blockDim.x) {
      const float4 xv = *(const float4*)(xr + f);
      const float4 t0 = *(const float4*)(mt + f), t1 = *(const float4*)(mt + D + f);
      const float4 d0 = *(const float4*)(md + f), d1 = *(const float4*)(md + D + f);
      const float4 b0 = *(const float4*)(mb + f), b1 = *(const float4*)(mb + D + f);
      const float xs[4] = {xv.x, xv.y, xv.z, xv.w};
      const float sc[4] = {t0.x + d0.x + b0.x, t0.y + d0.y + b0.y, t0.z + d0.z + b0.z, t0.w + d0.w + b0.w};
      const float sh[4] = {t1.x + d1.x + b1.x, t1.y + d1.y + b1.y, t1.z + d1.z + b1.z, t1.w + d1.w + b1.w};
      float y[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) y[e] = __bfloat162float(__float2bfloat16_rn(xs[e] * inv * (1.f + sc[e]) + sh[e]));
#pragma unroll
      for (int o = 0; o < 32; ++o) {
        if (FULL || o < A) {
          const uint2 wq = *(const uint2*)((const bf16*)h.w + (size_t)o * D + f);   // 4 bf16 of W_out row o
          acc[o] = fmaf(y[0], __uint_as_float(wq.x << 16), acc[o]);
          acc[o] = fmaf(y[1], __uint_as_float(wq.x & 0xFFFF0000u), acc[o]);
          acc[o] = fmaf(y[2], __uint_as_float(wq.y << 16), acc[o]);
          acc[o] = fmaf(y[3], __uint_as_float(wq.y & 0xFFFF0000u), acc[o]);
        }
      }
    }
    // warp: lane o ends with the warp's sum of output o (each step keeps half
    // of the outputs and adds the partner's half)
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      const bool up = (lane & off) != 0;
#pragma unroll
      for (int i = 0; i < off; ++i) {
        const float send = up ? acc[i] : acc[i + off];
        const float keep = up ? acc[i + off] : acc[i];
        acc[i] = keep + __shfl_xor_sync(0xffffffffu, send, off);
      }
    }
    red[warp][lane] = acc[0];
    __syncthreads();
    if (threadIdx.x < A) {
      float v = h.b[threadIdx.x];
#pragma unroll
      for (int w = 0; w < 8; ++w) v += red[w][threadIdx.x];
      h.v[(size_t)(b * a.H + j) * A + threadIdx.x] = v;
    }
    __syncthreads();   // red is reused by the next row
  }
  // the robot's last CTA to finish runs the tail
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int done = atomicAdd(h.cnt + b, 1);
    last = done == nb - 1;
    if (last) h.cnt[b] = 0;
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  tail_robot(a, b, sa);
}

cudaError_t launch_head_tail(const HeadArgs& h, const TailArgs& a, cudaStream_t st) {
  if (a.B <= 0) return cudaSuccess;
  const size_t smem = (size_t)a.H * a.A * sizeof(float);
  if (a.A > 32 || h.D % 4 || smem > 48 * 1024) return cudaErrorNotSupported;
  const int nb = (a.H + h.rows_per_cta - 1) / h.rows_per_cta;
  if (a.A == 32)
    return launch_kernel(head_tail_kernel<true>, dim3(a.B * nb), dim3(256), smem, st, 1, h, a);
  return launch_kernel(head_tail_kernel<false>, dim3(a.B * nb), dim3(256), smem, st, 1, h, a);
}

// Full-horizon denoising (the synchronous baseline): every slot takes the
// same Euler step a += dt v with dt = t_now - t_next (float32, read off the
// time grid like the rolling step's dt_j); nothing is released or shifted.
__global__ void denoise_tail_kernel(float* __restrict__ buffer, const float* __restrict__ vel, float* __restrict__ vel_out,
                                    int n, float t_now, float t_next) {
  pdl_trigger();
  pdl_wait();
  const float dt = __fsub_rn(t_now, t_next);
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    const float v = vel[i];
    buffer[i] = fmaf(dt, v, buffer[i]);
    if (vel_out) vel_out[i] = v;
  }
}

cudaError_t launch_denoise_tail(float* buffer, const float* vel, float* vel_out, int B, int H, int A, float t_now,
                                float t_next, cudaStream_t st) {
  const int n = B * H * A;
  if (n <= 0) return cudaSuccess;
  const int blocks = std::min((n + 255) / 256, 1024);
  return launch_kernel(denoise_tail_kernel, dim3(blocks), dim3(256), 0, st, 1, buffer, vel, vel_out, n, t_now, t_next);
}

// times[0..H-1] = t (the single flow time of a synchronous denoising pass).
__global__ void fill_times_kernel(float* __restrict__ times, int H, float t) {
  pdl_trigger();
  pdl_wait();
  for (int j = threadIdx.x; j < H; j += blockDim.x) times[j] = t;
}

cudaError_t launch_fill_times(float* times, int H, float t, cudaStream_t st) {
  return launch_kernel(fill_times_kernel, dim3(1), dim3(128), 0, st, 1, times, H, t);
}

// A fresh chunk: slot j of robot b receives the Gaussian action of index
// counters[b] + j, and the counter advances by H.
__global__ void chunk_noise_kernel(float* __restrict__ buffer, const uint64_t* __restrict__ seeds,
                                   uint64_t* __restrict__ counters, int H, int A) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int groups = (A + 3) / 4;
  const uint64_t n0 = counters[b];
  for (int i = threadIdx.x; i < H * groups; i += blockDim.x) {
    const int j = i / groups, g = i % groups;
    float z[4];
    action_noise4(seeds[b], n0 + (uint64_t)j, (uint32_t)g, z);
#pragma unroll
    for (int t = 0; t < 4; ++t)
      if (4 * g + t < A) buffer[((size_t)b * H + j) * A + 4 * g + t] = z[t];
  }
  __syncthreads();
  if (threadIdx.x == 0) counters[b] = n0 + (uint64_t)H;
}

cudaError_t launch_chunk_noise(float* buffer, const uint64_t* seeds, uint64_t* counters, int B, int H, int A,
                               cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  return launch_kernel(chunk_noise_kernel, dim3(B), dim3(128), 0, st, 1, buffer, seeds, counters, H, A);
}

cudaError_t init_simt_kernels() {
  const int att = (ATT_QT * 256 + 2 * ATT_KT * 256 + ATT_QT * ATT_KT) * (int)sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(attention_simt_kernel<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, att);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attention_simt_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, att);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tail_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 16384 * (int)sizeof(float));
  const int xa = (2 * 64 * 256 + 8 * 64) * (int)sizeof(float);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(fop_xattn_kernel<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize, xa);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(fop_xattn_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, xa);
  return e;
}

__global__ void reset_kernel(float* __restrict__ buffer, const uint64_t* __restrict__ seeds,
                             uint64_t* __restrict__ counters, int H, int A) {
  const int b = blockIdx.x;
  const int groups = (A + 3) / 4;
  for (int i = threadIdx.x; i < H * groups; i += blockDim.x) {
    const int j = i / groups, g = i % groups;
    float z[4];
    action_noise4(seeds[b], (uint64_t)j, (uint32_t)g, z);
#pragma unroll
    for (int t = 0; t < 4; ++t)
      if (4 * g + t < A) buffer[((size_t)b * H + j) * A + 4 * g + t] = z[t];
  }
  if (threadIdx.x == 0) counters[b] = (uint64_t)H;
}

cudaError_t launch_reset(float* buffer, const uint64_t* seeds, uint64_t* counters, int B, int H, int A,
                         cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  reset_kernel<<<B, 128, 0, st>>>(buffer, seeds, counters, H, A);
  return cudaGetLastError();
}

__global__ void delay_kernel(unsigned long long ns) {
  unsigned long long t0, t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  do {
    __nanosleep(10000);
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  } while (t - t0 < ns);
}

cudaError_t launch_delay(unsigned long long ns, cudaStream_t st) {
  delay_kernel<<<1, 1, 0, st>>>(ns);
  return cudaGetLastError();
}

__global__ void flip_kernel(int* s, CtxList f) {
  for (int i = threadIdx.x; i < f.n; i += blockDim.x) {
    s[2 * f.robot[i]] = f.slot[i];
    s[2 * f.robot[i] + 1] = f.len[i];
  }
}

cudaError_t launch_flip(int* ctx_state, const CtxList& f, cudaStream_t st) {
  if (f.n <= 0) return cudaSuccess;
  flip_kernel<<<1, 128, 0, st>>>(ctx_state, f);
  return cudaGetLastError();
}

// Context rows of the listed robots into their slots: source [L][src_n][Hkv]
// [P][row] with the list's robots at positions i0 .. i0 + f.n - 1 of each
// layer, destination [slot][L][Bmax][Hkv][Pmax][row] (16-byte words).
__global__ void ctx_scatter_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst0, uint4* __restrict__ dst1,
                                   int src_n, int i0, int Bmax, int Hkv, int P, int Pmax, int row_words, CtxList f) {
  const int z = blockIdx.y;                  // (l * f.n + i) * Hkv + g
  const int g = z % Hkv, li = z / Hkv;
  const int i = li % f.n, l = li / f.n;
  const size_t words = (size_t)P * row_words;
  const uint4* s = src + ((size_t)(l * src_n + i0 + i) * Hkv + g) * words;
  uint4* d = (f.slot[i] ? dst1 : dst0) + (((size_t)l * Bmax + f.robot[i]) * Hkv + g) * (size_t)Pmax * row_words;
  for (size_t w = (size_t)blockIdx.x * blockDim.x + threadIdx.x; w < words; w += (size_t)gridDim.x * blockDim.x)
    d[w] = s[w];
}

cudaError_t launch_ctx_scatter(const void* src, int src_n, int i0, void* dst0, void* dst1, int L, int Bmax, int Hkv,
                               int P, int Pmax, size_t row_bytes, const CtxList& f, cudaStream_t st) {
  if (f.n <= 0 || P <= 0) return cudaSuccess;
  if (row_bytes % 16 || ((uintptr_t)src | (uintptr_t)dst0 | (uintptr_t)dst1) % 16) return cudaErrorMisalignedAddress;
  const int row_words = (int)(row_bytes / 16);
  const size_t words = (size_t)P * row_words;
  dim3 grid((unsigned)std::min<size_t>((words + 255) / 256, 64), (unsigned)(L * f.n * Hkv));
  ctx_scatter_kernel<<<grid, 256, 0, st>>>((const uint4*)src, (uint4*)dst0, (uint4*)dst1, src_n, i0, Bmax, Hkv, P,
                                           Pmax, row_words, f);
  return cudaGetLastError();
}

}  // namespace ravel
