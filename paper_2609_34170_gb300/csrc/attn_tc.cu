// Grouped-query attention of the action slots on the 5th-generation tensor
// cores (tcgen05 + TMEM + TMA), flash-attention style.
//
// One CTA owns a tile of up to 128 query rows of one (robot b, KV head g)
// pair -- row r = t*G + hh is slot j0+t of query head g*G+hh -- and walks the
// pair's keys in chunks of 64: first the active VLM context's prefix
// (context slot, valid length read on the device), then the FOP tokens and
// the H action slots of this step (the QKV buffer).  Per chunk:
//   S = Q K^T        tcgen05.mma, M = 128 query rows, N = 64 keys, into TMEM
//   P = exp(S - m)   softmax warps: TMEM -> registers -> bf16 P back into TMEM
//   O += P V         tcgen05.mma, M = 128, N = head dim, K = 64 keys, O in TMEM
// Every operand is K-major with 128-byte swizzling; V is kept transposed
// (keys contiguous) for that: the context's V is transposed when a context
// is installed, and the step's own V by the QKV projection's epilogue.
// The online softmax rescales O in TMEM only when a row's running maximum
// grows by more than 2^8 (the kept maximum is exact for the final
// normalisation, so this is not an approximation).
// At batch 1 a (b, g) pair has only a few query tiles, so the key chunks are
// split over grid.z; the splits of a query tile form a thread-block cluster
// and rank q merges head-dim slice q of every split's partial.  Each split
// sends its rows' (m, l) and its output normalised by its own l, in bf16 (the
// precision of every activation between kernels of the bf16 path), by
// st.async straight into the owning rank's shared memory, overlaid on Q and
// the K ring, as soon as its own PV is done and every split's last S MMA has
// completed (a multicast tcgen05.commit on each split's "S done" barrier; a
// cluster barrier after all MMAs where the area reaches the V ring); an
// mbarrier at the owner counts the bytes.  Where that does not apply, the splits
// publish unnormalised fp32 partials through L2 and the cluster barrier.  The
// producer keeps the L2 warm a few prefix chunks ahead of its loads.
//
// Warp roles (192 threads): warp 0 TMA producer, warp 1 TMEM allocator + MMA
// issuer, warps 2..5 softmax / epilogue (warp w owns TMEM lanes 32*(w%4)..).
// Every wait is bounded (ERR_TIMEOUT, then unwind).
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "launch.h"
#include "tc_common.cuh"

namespace ravel {
namespace {

// warp 0: loads; warp 1: MMAs; warps 2-5: softmax (a thread per query row);
// warps 6-7 join only the merge of the key splits, so that each thread takes
// one (row, 8-column) item of a 64-row tile's slice instead of two
constexpr int AT_THREADS = 256;
constexpr int AT_BM = 128;
constexpr int AT_BKV = 64;
constexpr int AT_SMEM_MAX = 227 * 1024;
constexpr uint32_t AT_QBLK = AT_BM * 128;     // bytes of one 64-wide head-dim block of Q
constexpr uint32_t AT_KBLK = AT_BKV * 128;    // bytes of one 64-wide head-dim block of a K chunk

struct AtParams {
  int B, H, F, Hq, Hkv, G, hd, hdp;   // hdp: head dim rounded up to 16 (MMA N of P V)
  int TQ, q_tiles;
  int Pmax, n_pre, n_kv, splits;
  int layer, Bmax, mask_mode;
  int nblk, k_slots, v_slots;         // head-dim blocks of 64; K and V ring depths
  int xch;                            // splits > 1: partials through L2 (0) or shared memory, sent once every
                                      // split's MMAs are done (1: cluster barrier) or once every split's S
                                      // MMAs are done (2: the receive area lies in Q and the K ring)
  const int* ctx_state;
  bf16* out;
  int ld_out;
  float* ws_o;
  float* ws_ml;
  int* err;
  float scale_log2;                   // log2(e) / sqrt(hd)
};

// K and V chunks alike: [64 keys][64-wide head-dim block] boxes, 128-byte
// swizzled; V is the B operand of P V in its natural layout (MN-major)
struct AtMaps {
  CUtensorMap q, k, v, pk0, pk1, pv0, pv1;
};

// The idx-th chunk this CTA processes (prefix chunks past the valid prefix
// length are skipped), or -1.
__device__ __forceinline__ int chunk_at(const AtParams& p, int P, int c0, int c1, int idx) {
  const int pre_end = min(min(c1, p.n_pre), (P + AT_BKV - 1) / AT_BKV);
  const int npre = max(0, pre_end - c0);
  if (idx < npre) return c0 + idx;
  const int c = max(c0, p.n_pre) + (idx - npre);
  return c < c1 ? c : -1;
}


__device__ __forceinline__ int chunk_count(const AtParams& p, int P, int c0, int c1) {
  int n = 0;
  for (int c = c0; c < c1; ++c)
    if (!(c < p.n_pre && c * AT_BKV >= P)) ++n;
  return n;
}

// Rows of the split-KV combine: out = sum_s wgt[s] * O_s * inv over float4
// columns [c4b, c4e) of this thread's row, the SP partials of a column batch
// loaded together (one L2 round trip per batch).  src0 points at split 0 of
// the row; splits are sstride floats apart, float4 columns 512.
template <int SP>
__device__ __forceinline__ void combine_slice(const float* src0, size_t sstride, int c4b, int c4e, const float* wgt,
                                              float inv, bf16* orow, int hd, bool row_ok) {
  constexpr int KC = 32 / SP;
  for (int c4 = c4b; c4 < c4e; c4 += KC) {
    float4 x[SP][KC];
#pragma unroll
    for (int s2 = 0; s2 < SP; ++s2)
#pragma unroll
      for (int k = 0; k < KC; ++k)
        x[s2][k] = (c4 + k < c4e) ? __ldcg((const float4*)(src0 + (size_t)s2 * sstride + (size_t)(c4 + k) * 512))
                                  : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int k = 0; k < KC; ++k) {
      const int d = 4 * (c4 + k);
      if (c4 + k >= c4e || d >= hd) break;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int s2 = 0; s2 < SP; ++s2) {
        acc.x += wgt[s2] * x[s2][k].x;
        acc.y += wgt[s2] * x[s2][k].y;
        acc.z += wgt[s2] * x[s2][k].z;
        acc.w += wgt[s2] * x[s2][k].w;
      }
      if (row_ok)   // hd % 8 == 0 and d % 4 == 0: all four columns exist; 8-byte aligned
        *(uint2*)(orow + d) = make_uint2(pack_bf16x2(acc.x * inv, acc.y * inv), pack_bf16x2(acc.z * inv, acc.w * inv));
    }
  }
}

__device__ __forceinline__ uint4 lds_u4(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
  return v;
}
__device__ __forceinline__ float2 lds_f2(uint32_t a) {
  float2 v;
  asm volatile("ld.shared.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(a));
  return v;
}

// Merge of row r, head-dim group gq, over the SP splits' shares received in
// shared memory (O groups [s][g][row] of 8 bf16 from `og`, (m, l) [s][row]
// from `ml`, both shared-memory addresses of row 0): columns d0 + 8 gq .. +7
// of slice q, stored as bf16 (a group past hd is skipped).
//   O = sum_s 2^(m_s - M) l_s Ohat_s / sum_s 2^(m_s - M) l_s
template <int SP>
__device__ __forceinline__ void xch_combine_group(uint32_t og, uint32_t ml, int r, int ngs, int gq, int d0, int hd,
                                                  bf16* orow) {
  const int d = d0 + 8 * gq;
  if (d >= hd) return;
  float2 v[SP];
#pragma unroll
  for (int s2 = 0; s2 < SP; ++s2) v[s2] = lds_f2(ml + (uint32_t)(s2 * AT_BM + r) * 8u);
  uint4 u[SP];
#pragma unroll
  for (int s2 = 0; s2 < SP; ++s2) u[s2] = lds_u4(og + ((uint32_t)(s2 * ngs + gq) * AT_BM + r) * 16u);
  float M = -INFINITY;
#pragma unroll
  for (int s2 = 0; s2 < SP; ++s2) M = fmaxf(M, v[s2].x);
  float w[SP];
  float L = 0.f;
#pragma unroll
  for (int s2 = 0; s2 < SP; ++s2) {
    w[s2] = (v[s2].x == -INFINITY) ? 0.f : exp2f(v[s2].x - M) * v[s2].y;
    L += w[s2];
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  float acc[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) acc[k] = 0.f;
#pragma unroll
  for (int s2 = 0; s2 < SP; ++s2) {
    const float ws = w[s2] * inv;
    const uint32_t uu[4] = {u[s2].x, u[s2].y, u[s2].z, u[s2].w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      acc[2 * k] = fmaf(ws, __uint_as_float(uu[k] << 16), acc[2 * k]);
      acc[2 * k + 1] = fmaf(ws, __uint_as_float(uu[k] & 0xFFFF0000u), acc[2 * k + 1]);
    }
  }
  *(uint4*)(orow + d) = make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]),
                                   pack_bf16x2(acc[4], acc[5]), pack_bf16x2(acc[6], acc[7]));
}

__global__ void __launch_bounds__(AT_THREADS, 1) attn_tc_kernel(const __grid_constant__ AtMaps maps, AtParams p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned; derived from smem_raw by pointer arithmetic so that the
  // compiler keeps it (and everything indexed from it) in the shared window
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int SK = p.k_slots, SV = p.v_slots;   // K and V ring depths
  const uint32_t k_bytes = (uint32_t)p.nblk * AT_KBLK;   // one K or V chunk
  uint8_t* q_s = smem;
  uint8_t* kv_s = q_s + (size_t)p.nblk * AT_QBLK;   // K ring, then V ring
  uint8_t* v_ring = kv_s + (size_t)SK * k_bytes;
  uint64_t* bars = (uint64_t*)(v_ring + (size_t)SV * k_bytes);
  // K and V of a stage have their own barriers: K is released as soon as
  // S = Q K^T has been computed, V only after P V, so the next K load does
  // not wait for the softmax and the PV of the chunk it replaces
  uint64_t* q_full = bars;
  uint64_t* k_full = bars + 1;
  uint64_t* v_full = k_full + SK;
  uint64_t* k_empty = v_full + SV;
  uint64_t* v_empty = k_empty + SK;
  uint64_t* s_full = v_empty + SV;
  uint64_t* s_free = s_full + 2;
  uint64_t* p_full = s_free + 2;
  uint64_t* pv_done = p_full + 2;   // [2]: PV of chunk i completes pv_done[i & 1]
  uint64_t* rcv_bar = pv_done + 2;  // xch: every split's share of this rank has arrived
  uint64_t* sdone = rcv_bar + 1;    // xch 2: every split's last S MMA has completed (one arrival each)
  uint32_t* tmem_slot = (uint32_t*)(sdone + 1);
  int* flags = (int*)(tmem_slot + 1);   // [0] abort, [1] K issued, [2] K consumed, [3] V issued, [4] V consumed

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qt = blockIdx.x, bg = blockIdx.y, split = blockIdx.z;
  const int b = bg / p.Hkv, g = bg % p.Hkv;
  const int rows_per_robot = p.H + p.F;
  const int slot = p.ctx_state[2 * b];       // this robot's active context
  const int P = p.ctx_state[2 * b + 1];
  const int C = p.n_pre + p.n_kv;
  const int c0 = (int)((long)split * C / p.splits), c1 = (int)((long)(split + 1) * C / p.splits);
  const uint32_t ncols = (128 + p.hdp <= 256) ? 256u : 512u;
  const int ctx_z = (p.layer * p.Bmax + b) * p.Hkv + g;
  // query rows of this tile that hold a slot (rows 0 .. vrows-1)
  const int vrows = p.G * max(0, min(p.TQ, p.H - qt * p.TQ));
  // xch: per rank, [split][cps / 8][128 rows] groups of 8 bf16, then [split][128 rows] (m, l)
  const int cps = p.hdp / p.splits;

  pdl_trigger();
  if (P < 1 || P > p.Pmax) {   // uniform across the CTA: nothing allocated yet
    pdl_wait();
    if (threadIdx.x == 0) raise_error(p.err, ERR_PREFIX_LEN);
    return;
  }
  const int n = chunk_count(p, P, c0, c1);
  // the active context (slot, length and its prefix K/V) is fixed for the
  // whole step, so the first prefix chunks are fetched before the wait on the
  // previous kernel (the QKV projection)
  int npre = 0, c_next = c0;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < SK; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);   // released by the S commit
    }
    for (int s = 0; s < SV; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);   // released by the PV commit
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 128);
      mbar_init(&p_full[i], 128);
    }
    mbar_init(&pv_done[0], 1);
    mbar_init(&pv_done[1], 1);
    mbar_init(rcv_bar, 1);
    mbar_init(sdone, p.splits);
    flags[0] = flags[1] = flags[2] = flags[3] = flags[4] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    if (p.xch) mbar_expect_tx(rcv_bar, (uint32_t)(p.splits * vrows * (2 * cps + 8)));
  }
  // (xch 2) every split's barriers must exist before a peer targets them
  if (p.xch == 2) cluster_sync();
  const CUtensorMap* pk = slot ? &maps.pk1 : &maps.pk0;
  const CUtensorMap* pv = slot ? &maps.pv1 : &maps.pv0;
  // K and V of chunk c into stage s, each CTA loading its own copy (query
  // tiles of one (b, g) pair read the same chunk, which L2 serves to all)
  auto load_k = [&](int c, int s, uint64_t pol) {
    uint8_t* ks = kv_s + (size_t)s * k_bytes;
    mbar_expect_tx(&k_full[s], k_bytes);
    const bool pre = c < p.n_pre;
    const int cc = c - p.n_pre;
    const CUtensorMap* km = pre ? pk : &maps.k;
    const int ky = pre ? c * AT_BKV : g, kz = pre ? ctx_z : b * rows_per_robot + cc * AT_BKV;
    for (int blk = 0; blk < p.nblk; ++blk) tma_load_3d(km, &k_full[s], ks + (size_t)blk * AT_KBLK, blk * 64, ky, kz, pol);
  };
  auto load_v = [&](int c, int s, uint64_t pol) {
    uint8_t* vs = v_ring + (size_t)s * k_bytes;
    mbar_expect_tx(&v_full[s], k_bytes);
    const bool pre = c < p.n_pre;
    const int cc = c - p.n_pre;
    const CUtensorMap* vm = pre ? pv : &maps.v;
    const int vy = pre ? c * AT_BKV : g, vz = pre ? ctx_z : b * rows_per_robot + cc * AT_BKV;
    for (int blk = 0; blk < p.nblk; ++blk) tma_load_3d(vm, &v_full[s], vs + (size_t)blk * AT_KBLK, blk * 64, vy, vz, pol);
  };
  if (threadIdx.x == 0) {
    uint64_t pol_kv;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol_kv));
    for (; c_next < c1 && c_next < p.n_pre && npre < min(SK, SV); ++c_next) {
      if (c_next * AT_BKV >= P) continue;
      load_k(c_next, npre, pol_kv);
      load_v(c_next, npre, pol_kv);
      ++npre;
    }
    // and warm L2 with the prefix chunks that will refill those stages
    for (int k = 0; k < SK; ++k) {
      const int c = chunk_at(p, P, c0, c1, npre + k);
      if (c < 0 || c >= p.n_pre) break;
      for (int blk = 0; blk < p.nblk; ++blk) prefetch_l2_3d(pk, blk * 64, c * AT_BKV, ctx_z);
      prefetch_l2_3d(pv, c * AT_BKV, 0, ctx_z);
    }
  }
  // rows of the Q tile that no query fills are zeroed (their scores are unused)
  const int q_rows = p.TQ * p.G;
  if (q_rows < AT_BM) {
    for (int blk = 0; blk < p.nblk; ++blk) {
      uint4* z = (uint4*)(q_s + (size_t)blk * AT_QBLK + (size_t)q_rows * 128);
      for (int i = threadIdx.x; i < (AT_BM - q_rows) * 8; i += AT_THREADS) z[i] = make_uint4(0, 0, 0, 0);
    }
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
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
  const uint32_t o_col = 128;

  if (warp == 0) {
    if (lane == 0) {
      uint64_t pol_q, pol_kv;
      asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol_q));
      asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol_kv));
      mbar_expect_tx(q_full, (uint32_t)p.nblk * 128u * (uint32_t)q_rows);
      for (int blk = 0; blk < p.nblk; ++blk)
        tma_load_3d(&maps.q, q_full, q_s + (size_t)blk * AT_QBLK, blk * 64, g * p.G, b * rows_per_robot + qt * p.TQ,
                    pol_q);
      // K of chunk nk and V of chunk nv (nv <= nk), each as soon as its slot
      // is free; K may run ahead of V
      int nk = npre, nv = npre;
      unsigned long long t_last = globaltimer();
      bool ok = true;
      while (ok && (nk < n || nv < n)) {
        bool progress = false;
        if (nk < n && mbar_test_wait(&k_empty[nk % SK], ((uint32_t)(nk / SK) & 1u) ^ 1u)) {
          const int c = chunk_at(p, P, c0, c1, nk);
          load_k(c, nk % SK, c < p.n_pre ? pol_kv : pol_q);
          {   // keep the L2 warm 2 SK chunks ahead of the loads (prefix chunks only)
            const int cf = chunk_at(p, P, c0, c1, nk + 2 * SK);
            if (cf >= 0 && cf < p.n_pre) {
              for (int blk = 0; blk < p.nblk; ++blk) prefetch_l2_3d(pk, blk * 64, cf * AT_BKV, ctx_z);
              prefetch_l2_3d(pv, cf * AT_BKV, 0, ctx_z);
            }
          }
          ++nk;
          progress = true;
        }
        if (nv < nk && mbar_test_wait(&v_empty[nv % SV], ((uint32_t)(nv / SV) & 1u) ^ 1u)) {
          const int c = chunk_at(p, P, c0, c1, nv);
          load_v(c, nv % SV, c < p.n_pre ? pol_kv : pol_q);
          ++nv;
          progress = true;
        }
        if (progress) t_last = globaltimer();
        else if (globaltimer() - t_last > kTcTimeoutNs) ok = false;
      }
      if (!ok) flags[0] = 1;
      flags[1] = nk;
      flags[3] = nv;
    }
    __syncwarp();
    // xch 1: one arrival per thread on the cluster barrier that opens the
    // exchange (the softmax warps arrive once their last PV is complete)
    if (p.xch == 1) cluster_arrive_release();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc_s = idesc_bf16(AT_BM, AT_BKV);
      const uint32_t idesc_o = idesc_bf16_bmn(AT_BM, p.hdp);
      bool ok = mbar_wait(q_full, 0);
      // Issue S of the next chunk and PV of the oldest chunk whose P is ready,
      // whichever can go: PV(i) never waits for chunk i+1's K/V (that would
      // chain every chunk's load behind the previous PV).  S runs at most one
      // chunk ahead of PV (two S buffers in TMEM).
      int ns = 0, i = 0;   // next S, next PV
      bool sdone_sent = false;
      // xch 2: every split learns when this split's last S has completed
      // (its Q and K ring may then receive the partials of the merge)
      const uint16_t smask = (uint16_t)((1u << p.splits) - 1u);
      unsigned long long t_last = globaltimer();
      while (ok && i < n) {
        bool progress = false;
        if (ns < n && ns <= i + 1) {
          const int s = ns % SK;
          if (mbar_test_wait(&k_full[s], (uint32_t)(ns / SK) & 1u) &&
              (ns < 2 || mbar_test_wait(&s_free[ns & 1], (uint32_t)((ns >> 1) - 1) & 1u))) {
            tc_fence_after();
            const uint8_t* ks = kv_s + (size_t)s * k_bytes;
            for (int blk = 0; blk < p.nblk; ++blk) {
              const uint64_t ad = sw128_desc(smem_u32(q_s + (size_t)blk * AT_QBLK));
              const uint64_t bd = sw128_desc(smem_u32(ks + (size_t)blk * AT_KBLK));
#pragma unroll
              for (int k = 0; k < 4; ++k)
                umma_bf16(tmem + (uint32_t)(ns & 1) * AT_BKV, ad + 2 * k, bd + 2 * k, idesc_s,
                          (blk > 0 || k > 0) ? 1u : 0u);
            }
            umma_commit(&s_full[ns & 1]);
            umma_commit(&k_empty[s]);   // K of this stage is free once S is done
            ++ns;
            if (p.xch == 2 && ns == n) {
              umma_commit_mc(sdone, smask);
              sdone_sent = true;
            }
            progress = true;
          }
        }
        if (i < ns && mbar_test_wait(&p_full[i & 1], (uint32_t)(i >> 1) & 1u) &&
            mbar_test_wait(&v_full[i % SV], (uint32_t)(i / SV) & 1u)) {
          tc_fence_after();
          const int s = i % SV;
          // A = P from TMEM (the S tile's first 32 columns, two bf16 per column)
          const uint32_t pa = tmem + (uint32_t)(i & 1) * AT_BKV;
          // B = V [64 keys][hd], MN-major: 16 keys (two 8-row groups) per K step
          const uint64_t bd = sw128_mn_desc(smem_u32(v_ring + (size_t)s * k_bytes), AT_KBLK);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            umma_bf16_ts(tmem + o_col, pa + 8 * k, bd + 128 * k, idesc_o, (i > 0 || k > 0) ? 1u : 0u);
          umma_commit(&v_empty[s]);
          umma_commit(&pv_done[i & 1]);
          ++i;
          progress = true;
        }
        if (progress) {
          t_last = globaltimer();
        } else if (globaltimer() - t_last > kTcTimeoutNs) {
          ok = false;
        }
      }
      // (no chunk, or an abort: arrive all the same, once earlier MMAs are done)
      if (p.xch == 2 && !sdone_sent) umma_commit_mc(sdone, smask);
      if (!ok) flags[0] = 1;
      flags[2] = ns;   // chunks whose K arrival was consumed
      flags[4] = i;    // chunks whose V arrival was consumed
    }
    __syncwarp();
    if (p.xch == 1) cluster_arrive_release();
  } else if (warp >= 6) {
    // merge-only warps: one arrival on the cluster barrier that opens the exchange
    if (p.xch == 1) cluster_arrive_release();
  } else {
    // softmax / epilogue: thread owns query row r (TMEM lane r)
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(q4 * 32) << 16);
    const int t = r / p.G;
    const int j = qt * p.TQ + t;
    float m_used = -INFINITY, l = 0.f;   // running max (log2 domain, scaled) and sum of P
    bool ok = true;
    int i = 0;
    const float sl2 = p.scale_log2;
    for (int c = c0; c < c1 && ok; ++c) {
      if (c < p.n_pre && c * AT_BKV >= P) continue;
      ok = __all_sync(0xffffffffu, mbar_wait(&s_full[i & 1], (uint32_t)(i >> 1) & 1u));
      tc_fence_after();
      float sc[64];
      {
        uint32_t raw[64];
#pragma unroll
        for (int q = 0; q < 4; ++q) tmem_ld16_async(lane_base + (uint32_t)(i & 1) * AT_BKV + 16 * q, raw + 16 * q);
        tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 64; ++k) sc[k] = __uint_as_float(raw[k]);
      }
      tc_fence_before();
      mbar_arrive(&s_free[i & 1]);
      // keys of this chunk that exist (prefix shorter than the chunk, ragged
      // FOP + slot chunk) and, in the slot-isolated test mode, that are visible
      const int kk0 = (c < p.n_pre) ? c * AT_BKV : (c - p.n_pre) * AT_BKV;
      const int kvalid = (c < p.n_pre) ? P - kk0 : rows_per_robot - kk0;
      const bool iso = (p.mask_mode == 1) && (c >= p.n_pre) && (kk0 < p.H);
      // (two compact loops: this code runs cold at batch 1, where each
      // instruction fetched costs more than it does)
      if (kvalid < AT_BKV) {
#pragma unroll
        for (int k = 0; k < 64; ++k) sc[k] = k < kvalid ? sc[k] : -INFINITY;
      }
      if (iso) {
#pragma unroll
        for (int k = 0; k < 64; ++k)
          if (kk0 + k < p.H && kk0 + k != j) sc[k] = -INFINITY;
      }
      float m8[8];
#pragma unroll
      for (int a = 0; a < 8; ++a)
        m8[a] = fmaxf(fmaxf(fmaxf(sc[8 * a], sc[8 * a + 1]), fmaxf(sc[8 * a + 2], sc[8 * a + 3])),
                      fmaxf(fmaxf(sc[8 * a + 4], sc[8 * a + 5]), fmaxf(sc[8 * a + 6], sc[8 * a + 7])));
      const float mx = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                             fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7]))) * sl2;
      const float m_new = fmaxf(m_used, mx);
      const bool need = m_new > m_used + 8.f;
      if (i > 0 && __any_sync(0xffffffffu, need)) {
        // O must hold PV of every earlier chunk before it is rescaled
        ok = __all_sync(0xffffffffu, mbar_wait(&pv_done[(i - 1) & 1], (uint32_t)((i - 1) >> 1) & 1u)) && ok;
        tc_fence_after();
        const float alpha = need ? exp2f(m_used - m_new) : 1.f;   // exp2(-inf) = 0
        for (int cb = 0; cb < p.hdp; cb += 16) {
          float o[16];
          tmem_ld16(lane_base + o_col + cb, o);
#pragma unroll
          for (int q = 0; q < 16; ++q) o[q] *= alpha;
          tmem_st16(lane_base + o_col + cb, o);
        }
        tmem_wait_st();
        l *= alpha;
      }
      if (need) m_used = m_new;
      const float nb = (m_used == -INFINITY) ? 0.f : -m_used;
      // P (bf16) overwrites the first 32 columns of this chunk's S tile: S of
      // chunk i + 2 reuses the tile only after PV of chunk i has been issued,
      // and the tensor pipe runs them in order
      const uint32_t prow = lane_base + (uint32_t)(i & 1) * AT_BKV;
      float ls[8];
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        uint32_t w[16];
#pragma unroll
        for (int ch = 0; ch < 4; ++ch) {
          float e[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) e[q] = fast_exp2(fmaf(sc[32 * h2 + 8 * ch + q], sl2, nb));
          ls[4 * h2 + ch] = ((e[0] + e[1]) + (e[2] + e[3])) + ((e[4] + e[5]) + (e[6] + e[7]));
#pragma unroll
          for (int q = 0; q < 4; ++q) w[4 * ch + q] = pack_bf16x2(e[2 * q], e[2 * q + 1]);
        }
        tmem_st16u(prow + 16 * h2, w);
      }
      tmem_wait_st();
      l += ((ls[0] + ls[1]) + (ls[2] + ls[3])) + ((ls[4] + ls[5]) + (ls[6] + ls[7]));
      tc_fence_before();
      mbar_arrive(&p_full[i & 1]);
      ++i;
    }
    if (ok && n > 0) {
      ok = __all_sync(0xffffffffu, mbar_wait(&pv_done[(n - 1) & 1], (uint32_t)((n - 1) >> 1) & 1u));
      tc_fence_after();
    }
    if (!ok && lane == 0) flags[0] = 1;
    if (p.xch == 1) {
      // past this barrier every split of the cluster has finished its MMAs
      // (its Q and rings may be overwritten) and armed its receive barrier;
      // every thread arrives exactly once, whatever happened before
      cluster_arrive_release();
      cluster_wait_acquire();
    } else if (p.xch == 2) {
      // every split's S MMAs are done: their Q and K rings, where the
      // partials land, are no longer read
      const bool okd = __all_sync(0xffffffffu, mbar_wait_cluster(sdone, 0));
      if (!okd && lane == 0) flags[0] = 1;
    }
    if (p.splits == 1) {
      // O / l as bf16: this thread stages its row in the rings (every chunk
      // has been consumed and every MMA has completed, so nothing writes
      // there any more; rows padded by 16 bytes so that the warp's 16-byte
      // stores hit distinct banks) and hands it to the bulk copy engine as one
      // contiguous hd-wide output row
      const float inv = (l > 0.f && n > 0) ? 1.f / l : 0.f;
      const int rbytes = ((2 * p.hdp + 63) & ~63) + 16;   // whole 32-column writes, + 16 against bank conflicts
      uint8_t* srow = kv_s + (size_t)r * rbytes;
      for (int cb = 0; cb < p.hdp; cb += 32) {
        uint32_t raw[32];
        tmem_ld16_async(lane_base + o_col + cb, raw);
        tmem_ld16_async(lane_base + o_col + cb + 16, raw + 16);
        tmem_wait_ld();
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint4 w;
          w.x = pack_bf16x2(__uint_as_float(raw[8 * q]) * inv, __uint_as_float(raw[8 * q + 1]) * inv);
          w.y = pack_bf16x2(__uint_as_float(raw[8 * q + 2]) * inv, __uint_as_float(raw[8 * q + 3]) * inv);
          w.z = pack_bf16x2(__uint_as_float(raw[8 * q + 4]) * inv, __uint_as_float(raw[8 * q + 5]) * inv);
          w.w = pack_bf16x2(__uint_as_float(raw[8 * q + 6]) * inv, __uint_as_float(raw[8 * q + 7]) * inv);
          *(uint4*)(srow + (cb / 8 + q) * 16) = w;
        }
      }
      const int t = r / p.G, jj = qt * p.TQ + t;
      if (r < q_rows && jj < p.H) {
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        bulk_copy_s2g(p.out + (size_t)(b * p.H + jj) * p.ld_out + (size_t)(g * p.G + r % p.G) * p.hd, srow,
                      (uint32_t)(2 * p.hd));
        bulk_commit();
        bulk_wait_read<0>();   // read out before the shared memory goes away
      }
    } else if (p.xch) {
      // rows holding a slot: (m, l) to every rank; O / l as bf16, head-dim
      // slice q to rank q, starting with this split's own slice so that the
      // splits send to different ranks at any moment.  The TMEM loads are
      // warp-collective: every lane runs them, only rows that hold a slot send.
      const bool snd = r < vrows;
      const bool has = n > 0 && l > 0.f;
      const float inv = has ? 1.f / l : 0.f;
      const int ngs = cps / 8;
      const uint32_t base = smem_u32(smem);
      const uint32_t o0 = base + (uint32_t)(split * ngs * AT_BM + r) * 16u;
      const uint32_t bar0 = smem_u32(rcv_bar);
      if (snd) {
        const uint32_t ml0 = base + (uint32_t)(p.splits * ngs * AT_BM) * 16u + (uint32_t)(split * AT_BM + r) * 8u;
        const float m_s = has ? m_used : -INFINITY, l_s = has ? l : 0.f;
        for (int q = 0; q < p.splits; ++q) st_async_f2(mapa_shared(ml0, (uint32_t)q), m_s, l_s, mapa_shared(bar0, (uint32_t)q));
      }
      // 32 columns per TMEM load (16 where hdp is not a multiple of 32), the
      // next load in flight while this one goes out
      const int cw = (p.hdp % 32 == 0) ? 32 : 16;
      const int nch = p.hdp / cw;
      int ch = (split * cps) / cw;
      uint32_t cur[32];
      if (cw == 32) tmem_ld32_async(lane_base + o_col + 32 * ch, cur);
      else tmem_ld16_async(lane_base + o_col + 16 * ch, cur);
      tmem_wait_ld();
      tmem_reg_fence16(cur);
      tmem_reg_fence16(cur + 16);
      for (int jj = 0; jj < nch; ++jj) {
        const int chn = ch + 1 == nch ? 0 : ch + 1;
        uint32_t nxt[32];
        if (jj + 1 < nch) {
          if (cw == 32) tmem_ld32_async(lane_base + o_col + 32 * chn, nxt);
          else tmem_ld16_async(lane_base + o_col + 16 * chn, nxt);
        }
        if (snd) {
          // groups of 8 columns: group g of the row goes to rank g / ngs, slot
          // g % ngs there (one division per chunk, then a running count)
          const int gidx0 = (cw / 8) * ch;
          int dst = gidx0 / ngs, gl = gidx0 - dst * ngs;
          auto send8 = [&](int h) {
            uint4 w;
            w.x = pack_bf16x2(__uint_as_float(cur[8 * h]) * inv, __uint_as_float(cur[8 * h + 1]) * inv);
            w.y = pack_bf16x2(__uint_as_float(cur[8 * h + 2]) * inv, __uint_as_float(cur[8 * h + 3]) * inv);
            w.z = pack_bf16x2(__uint_as_float(cur[8 * h + 4]) * inv, __uint_as_float(cur[8 * h + 5]) * inv);
            w.w = pack_bf16x2(__uint_as_float(cur[8 * h + 6]) * inv, __uint_as_float(cur[8 * h + 7]) * inv);
            if (!has) w = make_uint4(0u, 0u, 0u, 0u);   // no key: the accumulator was never written
            st_async_u4(mapa_shared(o0 + (uint32_t)gl * (AT_BM * 16), (uint32_t)dst), w,
                        mapa_shared(bar0, (uint32_t)dst));
            const bool wrap = ++gl == ngs;
            gl = wrap ? 0 : gl;
            dst += wrap ? 1 : 0;
          };
          send8(0);
          send8(1);
          if (cw == 32) {
            send8(2);
            send8(3);
          }
        }
        if (jj + 1 < nch) {
          tmem_wait_ld();
          tmem_reg_fence16(nxt);
          tmem_reg_fence16(nxt + 16);
#pragma unroll
          for (int k = 0; k < 32; ++k) cur[k] = nxt[k];
        }
        ch = chn;
      }
    } else {
      // unnormalised partial O as [ti][d/4][row][4] (a warp stores one
      // contiguous 512-byte run per 4 columns), plus this split's (m, l)
      const size_t ti = ((size_t)bg * gridDim.x + qt) * p.splits + split;
      float* dst = p.ws_o + ti * (size_t)(p.hdp / 4) * 512 + (size_t)r * 4;
      for (int cb = 0; cb < p.hdp; cb += 64) {   // up to four TMEM loads in flight, one wait
        const int nq = min(4, (p.hdp - cb) / 16);
        uint32_t raw[64];
#pragma unroll
        for (int q = 0; q < 4; ++q)
          if (q < nq) tmem_ld16_async(lane_base + o_col + cb + 16 * q, raw + 16 * q);
        tmem_wait_ld();
#pragma unroll
        for (int q = 0; q < 16; ++q)
          if (q < 4 * nq)
            __stcg((float4*)(dst + (size_t)(cb / 4 + q) * 512),
                   (n > 0) ? make_float4(__uint_as_float(raw[4 * q]), __uint_as_float(raw[4 * q + 1]),
                                         __uint_as_float(raw[4 * q + 2]), __uint_as_float(raw[4 * q + 3]))
                           : make_float4(0.f, 0.f, 0.f, 0.f));
      }
      __stcg(p.ws_ml + (ti * 2) * AT_BM + r, (n > 0) ? m_used : -INFINITY);
      __stcg(p.ws_ml + (ti * 2 + 1) * AT_BM + r, (n > 0) ? l : 0.f);
      __threadfence();
    }
  }
  tc_fence_before();
  cta_sync();
  if (flags[0]) {
    if (threadIdx.x == 0) {
      for (int i = flags[2]; i < flags[1]; ++i) mbar_wait(&k_full[i % SK], (uint32_t)(i / SK) & 1u);
      for (int i = flags[4]; i < flags[3]; ++i) mbar_wait(&v_full[i % SV], (uint32_t)(i / SV) & 1u);
      raise_error(p.err, ERR_TIMEOUT);
    }
    cta_sync();
  }
  if (p.xch) {
    // Rank q merges head-dim columns [q*cps, (q+1)*cps) of its rows once every
    // split's share has arrived (the wait also keeps this CTA alive until no
    // store into its shared memory is in flight):
    //   O = sum_s 2^(m_s - M) l_s Ohat_s / sum_s 2^(m_s - M) l_s,  Ohat_s = O_s / l_s.
    // Every warp takes part (the producer and MMA warps are idle by now):
    // work item (row r, 8-column group gq) of this rank's slice.
    {
      const bool ok = __all_sync(0xffffffffu, mbar_wait_cluster(rcv_bar, 0));
      if (!ok) {
        if (lane == 0) raise_error(p.err, ERR_TIMEOUT);
      } else {
        const int ngs = cps / 8, items = vrows * ngs;
        const uint32_t og = smem_u32(smem);
        const uint32_t ml = og + (uint32_t)(p.splits * ngs * AT_BM) * 16u;
        for (int it = threadIdx.x; it < items; it += AT_THREADS) {
          const int r = it % vrows, gq = it / vrows;
          const int t = r / p.G, hh = r % p.G;
          const int j = qt * p.TQ + t;
          bf16* orow = p.out + (size_t)(b * p.H + j) * p.ld_out + (size_t)(g * p.G + hh) * p.hd;
          switch (p.splits) {
            case 2: xch_combine_group<2>(og, ml, r, ngs, gq, split * cps, p.hd, orow); break;
            case 4: xch_combine_group<4>(og, ml, r, ngs, gq, split * cps, p.hd, orow); break;
            case 8: xch_combine_group<8>(og, ml, r, ngs, gq, split * cps, p.hd, orow); break;
            default: xch_combine_group<16>(og, ml, r, ngs, gq, split * cps, p.hd, orow); break;
          }
        }
      }
    }
  } else if (p.splits > 1) {
    // The key splits of this query tile form a cluster: once every split has
    // published its (O, m, l), rank q merges head-dim columns
    // [q*hdp/S, (q+1)*hdp/S):  O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s.
    cluster_sync();
    if (warp >= 2 && warp < 6) {
      const int r = (warp & 3) * 32 + lane;
      const int Sp = p.splits;
      const int cps = p.hdp / Sp;   // a multiple of 4
      const int rank = (int)cluster_ctarank();
      const size_t t0 = ((size_t)bg * gridDim.x + qt) * Sp;
      float wgt[16];
      float M = -INFINITY, L = 0.f;
#pragma unroll
      for (int s2 = 0; s2 < 16; ++s2) {
        wgt[s2] = -INFINITY;
        if (s2 >= Sp) continue;
        wgt[s2] = __ldcg(p.ws_ml + ((t0 + s2) * 2) * AT_BM + r);
        M = fmaxf(M, wgt[s2]);
      }
#pragma unroll
      for (int s2 = 0; s2 < 16; ++s2) {
        if (s2 >= Sp) break;
        const float l_s = __ldcg(p.ws_ml + ((t0 + s2) * 2 + 1) * AT_BM + r);
        wgt[s2] = (wgt[s2] == -INFINITY) ? 0.f : exp2f(wgt[s2] - M);
        L += wgt[s2] * l_s;
      }
      const float inv = L > 0.f ? 1.f / L : 0.f;
      const int t = r / p.G, hh = r % p.G;
      const int j = qt * p.TQ + t;
      const bool row_ok = (r < p.TQ * p.G) && (j < p.H);
      bf16* orow = p.out + (size_t)(b * p.H + j) * p.ld_out + (size_t)(g * p.G + hh) * p.hd;
      const float* src0 = p.ws_o + t0 * (size_t)(p.hdp / 4) * 512 + (size_t)r * 4;
      const size_t sstride = (size_t)(p.hdp / 4) * 512;
      const int c4b = rank * cps / 4, c4e = (rank + 1) * cps / 4;
      switch (Sp) {
        case 2: combine_slice<2>(src0, sstride, c4b, c4e, wgt, inv, orow, p.hd, row_ok); break;
        case 4: combine_slice<4>(src0, sstride, c4b, c4e, wgt, inv, orow, p.hd, row_ok); break;
        case 8: combine_slice<8>(src0, sstride, c4b, c4e, wgt, inv, orow, p.hd, row_ok); break;
        default: combine_slice<16>(src0, sstride, c4b, c4e, wgt, inv, orow, p.hd, row_ok); break;
      }
    }
  }
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols) : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;
int g_attn_max_cluster = 8;   // largest power-of-two cluster of key splits

cudaError_t enc3(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t s1_bytes,
                 uint64_t s2_bytes, uint32_t b0, uint32_t b1, uint32_t b2) {
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {s1_bytes, s2_bytes};
  cuuint32_t box[3] = {b0, b1, b2};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace

cudaError_t init_attention_tc() {
  if (!g_enc) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess) return e;
    if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorSymbolNotFound;
    g_enc = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  }
  cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, AT_SMEM_MAX);
  if (e != cudaSuccess) return e;
  if (cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 1;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 16;
    cfg.gridDim = dim3(1, 1, 16);
    cfg.blockDim = dim3(AT_THREADS);
    cfg.dynamicSmemBytes = AT_SMEM_MAX;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, attn_tc_kernel, &cfg) == cudaSuccess && n > 0) g_attn_max_cluster = 16;
  }
  cudaGetLastError();
  return cudaSuccess;
}

bool attention_tc_supported(int hd, int G) { return hd % 8 == 0 && hd <= 256 && G >= 1 && G <= 128; }

cudaError_t launch_attention_tc(const AttnTcArgs& a, cudaStream_t st) {
  if (!g_enc) return cudaErrorInitializationError;
  AtParams p{};
  p.B = a.B; p.H = a.H; p.F = a.F; p.Hq = a.Hq; p.Hkv = a.Hkv; p.G = a.Hq / a.Hkv; p.hd = a.hd;
  p.hdp = (a.hd + 15) / 16 * 16;
  const int tq_max = AT_BM / p.G;
  p.q_tiles = (a.H + tq_max - 1) / tq_max;
  p.TQ = (a.H + p.q_tiles - 1) / p.q_tiles;
  p.Pmax = a.Pmax;
  p.n_pre = (a.Pmax + AT_BKV - 1) / AT_BKV;
  p.n_kv = (a.H + a.F + AT_BKV - 1) / AT_BKV;
  p.layer = a.layer; p.Bmax = a.Bmax; p.mask_mode = a.mask_mode;
  p.nblk = (a.hd + 63) / 64;
  p.ctx_state = a.ctx_state;
  p.out = (bf16*)a.out; p.ld_out = a.ld_out;
  p.err = a.err;
  p.scale_log2 = 1.4426950408889634f / sqrtf((float)a.hd);
  const int C = p.n_pre + p.n_kv;
  // when the keys will be split (the grid leaves most SMs idle), query tiles
  // of 64 rows: the merge moves every split's rows x hd partial between the
  // SMs of the cluster, so its time grows with the rows of a tile, while the
  // MMAs (always 128 rows) and the key loads of a split do not; the grid
  // (at up to 8 splits) stays within half the SMs, which are free while the
  // previous kernel still holds the rest, so that every CTA starts early
  {
    const int tq_small = std::max(1, 64 / p.G);
    const int qt_small = (a.H + tq_small - 1) / tq_small;
    if (p.q_tiles * a.B * a.Hkv * 2 <= a.num_sms && tq_small < p.TQ && qt_small * a.B * a.Hkv * 8 <= a.num_sms / 2 &&
        (C + 1) / 2 >= 2) {
      p.q_tiles = qt_small;
      p.TQ = (a.H + qt_small - 1) / qt_small;
    }
  }
  const int nctas = p.q_tiles * a.B * a.Hkv;
  // split the key chunks only when the (b, g, q-tile) grid leaves most SMs
  // idle; about two chunks per split so S(i+1) overlaps the softmax of i
  // the splits of a query tile form one cluster (power of two, <= 16) whose
  // head-dim slices are multiples of 4 columns
  int splits = 1;
  if (nctas * 2 <= a.num_sms) {
    const int cap = std::min({(C + 1) / 2, std::max(1, a.num_sms / nctas), g_attn_max_cluster});
    while (splits * 2 <= cap && (p.hdp / (splits * 2)) % 4 == 0 &&
           (size_t)(splits * 2) * nctas * AT_BM * (p.hdp + 2) * 4 <= a.ws_bytes)
      splits *= 2;
  }
  p.splits = splits;
  p.ws_o = a.ws;
  p.ws_ml = a.ws + (size_t)splits * nctas * AT_BM * p.hdp;
  // partials through shared memory: whole 8-column bf16 groups per rank
  // slice, and the receive area (O groups + (m, l) of every split) within
  // Q + the rings (checked below)
  p.xch = splits > 1 && (p.hdp / splits) % 8 == 0 ? 1 : 0;
  // K slots: as many whole K + V stages as fit (<= 4); V slots: the K count
  // plus what the remaining bytes hold (<= 2 more): K is free again as soon
  // as S = Q K^T is done, V only after P V, so V needs the depth
  const size_t k_bytes = (size_t)p.nblk * AT_KBLK;
  const size_t stage = 2 * k_bytes;
  const size_t fixed = 1024 + (size_t)p.nblk * AT_QBLK + 512;
  if (fixed + stage > (size_t)AT_SMEM_MAX) return cudaErrorInvalidConfiguration;
  const int sk = (int)std::min<size_t>(4, (AT_SMEM_MAX - fixed) / stage);
  const int sv = sk + (int)std::min<size_t>(2, (AT_SMEM_MAX - fixed - sk * stage) / k_bytes);
  const size_t rings = (size_t)(sk + sv) * k_bytes;
  // the epilogue stages 128 bf16 rows of O in the rings and stores them with
  // 16-byte writes
  if ((size_t)AT_BM * (size_t)(((2 * p.hdp + 63) & ~63) + 16) > rings) return cudaErrorInvalidConfiguration;
  if (a.ld_out % 8 != 0 || ((uintptr_t)a.out & 15u) != 0) return cudaErrorMisalignedAddress;
  p.k_slots = sk;
  p.v_slots = sv;
  const size_t smem = fixed + rings;
  if (p.xch && (size_t)AT_BM * p.hdp * 2 + (size_t)splits * AT_BM * 8 > (size_t)p.nblk * AT_QBLK + rings) p.xch = 0;
  // the receive area within Q and the K ring (free once S is done): send
  // without waiting for the other splits' PV
  if (p.xch && (size_t)AT_BM * p.hdp * 2 + (size_t)splits * AT_BM * 8 <= (size_t)p.nblk * AT_QBLK + (size_t)sk * k_bytes)
    p.xch = 2;

  AtMaps m;
  const int hd = a.hd, rpr = a.H + a.F;
  const uint64_t rows = (uint64_t)a.B * rpr;
  cudaError_t e = enc3(&m.q, a.qkv, hd, a.Hq, rows, (uint64_t)hd * 2, (uint64_t)a.ld_qkv * 2, 64, p.G, p.TQ);
  if (e == cudaSuccess)
    e = enc3(&m.k, (const bf16*)a.qkv + (size_t)a.Hq * hd, hd, a.Hkv, rows, (uint64_t)hd * 2, (uint64_t)a.ld_qkv * 2,
             64, 1, AT_BKV);
  if (e == cudaSuccess)
    e = enc3(&m.v, (const bf16*)a.qkv + (size_t)(a.Hq + a.Hkv) * hd, hd, a.Hkv, rows, (uint64_t)hd * 2,
             (uint64_t)a.ld_qkv * 2, 64, 1, AT_BKV);
  const uint64_t zc = (uint64_t)(a.layers * a.Bmax * a.Hkv);
  for (int s = 0; s < 2 && e == cudaSuccess; ++s) {
    e = enc3(s ? &m.pk1 : &m.pk0, a.ctx_k[s], hd, a.Pmax, zc, (uint64_t)hd * 2, (uint64_t)a.Pmax * hd * 2, 64,
             AT_BKV, 1);
    if (e == cudaSuccess)
      e = enc3(s ? &m.pv1 : &m.pv0, a.ctx_v[s], hd, a.Pmax, zc, (uint64_t)hd * 2, (uint64_t)a.Pmax * hd * 2, 64,
               AT_BKV, 1);
  }
  if (e != cudaSuccess) return e;
  dim3 grid(p.q_tiles, a.B * a.Hkv, splits);
  e = launch_kernel_cluster(attn_tc_kernel, grid, dim3(AT_THREADS), smem, st, dim3(1, 1, splits), m, p);
  if (a.n_launched) ++*a.n_launched;
  return e;
}

}  // namespace ravel
