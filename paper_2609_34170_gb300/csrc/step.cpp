// Step plan: allocation, weight packing and the kernel sequence of one
// rolling action-expert step.
#include "step.h"

#include "launch.h"

#include <cstdio>
#include <algorithm>
#include <cmath>
#include <cstring>

namespace ravel {

bool validate_config(const ravel_config& c, std::string* why) {
  auto bad = [&](const char* m) {
    *why = m;
    return false;
  };
  if (c.layers < 1 || c.width < 8 || c.width % 8 || c.width > 4096)
    return bad("layers >= 1 and a width that is a multiple of 8 in [8, 4096] are required");
  if (c.n_q_heads < 1 || c.n_kv_heads < 1 || c.n_q_heads % c.n_kv_heads)
    return bad("n_q_heads must be a positive multiple of n_kv_heads");
  if (c.head_dim < 8 || c.head_dim > 256 || c.head_dim % 8) return bad("head_dim must be a multiple of 8 in [8, 256]");
  if (c.mlp_dim < 64 || c.mlp_dim % 64) return bad("mlp_dim must be a positive multiple of 64");
  if (c.slots < 1 || c.action_dim < 1 || (long)c.slots * c.action_dim > 16384)
    return bad("slots >= 1, action_dim >= 1 and slots * action_dim <= 16384 are required");
  if (c.max_prefix < 1 || c.fop_tokens < 0 || c.max_batch < 1) return bad("max_prefix, max_batch >= 1, fop_tokens >= 0");
  if (c.dtype != RAVEL_FP32 && c.dtype != RAVEL_BF16) return bad("dtype must be RAVEL_FP32 or RAVEL_BF16");
  if (c.mask_mode != RAVEL_MASK_FULL && c.mask_mode != RAVEL_MASK_SLOT_ISOLATED) return bad("unknown mask_mode");
  if (c.per_robot_times != 0 && c.per_robot_times != 1) return bad("per_robot_times must be 0 or 1");
  if (c.fop_adapter_every < 0 || c.fop_adapter_every > c.layers)
    return bad("fop_adapter_every must be 0 or in [1, layers]");
  if (c.fop_adapter_every > 0 && (c.fop_tokens < 1 || c.fop_tokens > 64))
    return bad("FOP adapters need 1 <= fop_tokens <= 64");
  return true;
}

static cudaError_t dalloc(StepPlan* p, void** ptr, size_t bytes) {
  *ptr = nullptr;
  if (bytes == 0) bytes = 16;
  cudaError_t e = cudaMalloc(ptr, bytes);
  if (e == cudaSuccess) {
    p->allocs.push_back(*ptr);
    e = cudaMemset(*ptr, 0, bytes);
  }
  return e;
}

void plan_destroy(StepPlan* p) {
  for (void* a : p->allocs) cudaFree(a);
  p->allocs.clear();
}

namespace {

struct Packer {
  StepPlan* p;
  const ravel_weights* w;
  float* staging;
  cudaError_t err = cudaSuccess;

  // device fp32 view of `n` floats at src (host or device)
  const float* view(const float* src, size_t n) {
    if (w->on_device) return src;
    if (err == cudaSuccess) err = cudaMemcpy(staging, src, n * sizeof(float), cudaMemcpyHostToDevice);
    return staging;
  }
  // dst = src^T ([K, N] -> [N, K]) in the plan's dtype
  void transpose(const float* src, int K, int N, void* dst, int interleave = 0, int off = 0) {
    const float* s = view(src, (size_t)K * N);
    if (err == cudaSuccess) err = launch_pack_transpose(s, K, N, dst, p->dt, interleave, off, 0);
    if (err == cudaSuccess) err = cudaDeviceSynchronize();
  }
  void copy_f32(const float* src, size_t n, float* dst) {
    if (err != cudaSuccess) return;
    err = cudaMemcpy(dst, src, n * sizeof(float), w->on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice);
  }
};

}  // namespace

ravel_status plan_create(StepPlan* p, const ravel_config& c, const ravel_weights& w, std::string* errs) {
  const ravel_weights* wp = &w;
  const float* req[] = {w.t_w1, w.t_b1, w.t_w2, w.t_b2, w.d_w1, w.d_b1, w.d_w2, w.d_b2, w.mod_w, w.mod_b,
                        w.in_w, w.in_b, w.fop_gamma, w.w_qkv, w.w_o, w.w_gate, w.w_up, w.w_down, w.out_w, w.out_b};
  for (const float* q : req)
    if (!q) {
      *errs = "a weight pointer is null";
      return RAVEL_EINVAL;
    }
  if (c.fop_adapter_every > 0 && (!w.a_gamma || !w.a_zgamma || !w.a_wq || !w.a_wkv || !w.a_wo || !w.a_gate)) {
    *errs = "an adapter weight pointer is null";
    return RAVEL_EINVAL;
  }
  p->cfg = c;
  p->dt = c.dtype == RAVEL_BF16 ? DT_BF16 : DT_F32;
  p->esize = c.dtype == RAVEL_BF16 ? 2 : 4;
  const size_t es = p->esize;
  const int D = c.width, L = c.layers, H = c.slots, A = c.action_dim, F = c.fop_tokens, Fm = c.mlp_dim;
  const int Bm = c.max_batch;
  p->nqkv = (c.n_q_heads + 2 * c.n_kv_heads) * c.head_dim;
  p->qdim = c.n_q_heads * c.head_dim;
  p->mod_dim = 4 * L * D + 2 * D;
  const size_t DD = (size_t)D * D;

  cudaError_t e = init_simt_kernels();
#define AL(ptr, bytes)                                      \
  do {                                                      \
    if (e == cudaSuccess) e = dalloc(p, (void**)&(ptr), (bytes)); \
  } while (0)
  AL(p->t_w1, DD * es); AL(p->t_w2, DD * es); AL(p->d_w1, DD * es); AL(p->d_w2, DD * es);
  AL(p->mod_w, (size_t)p->mod_dim * D * es);
  AL(p->w_qkv, (size_t)L * p->nqkv * D * es);
  AL(p->w_o, (size_t)L * D * p->qdim * es);
  AL(p->w_gu, (size_t)L * 2 * Fm * D * es);
  AL(p->w_down, (size_t)L * D * Fm * es);
  AL(p->out_w, (size_t)A * D * es);
  AL(p->t_b1, D * 4); AL(p->t_b2, D * 4); AL(p->d_b1, D * 4); AL(p->d_b2, D * 4);
  AL(p->mod_b, (size_t)p->mod_dim * 4);
  AL(p->in_w, (size_t)A * D * 4); AL(p->in_b, D * 4);
  AL(p->fop_gamma, (size_t)L * D * 4);
  AL(p->out_b, A * 4);
  const size_t ctx_bytes = (size_t)L * Bm * c.n_kv_heads * c.max_prefix * c.head_dim * es;
  for (int s = 0; s < 2; ++s) {
    AL(p->ctx_k[s], ctx_bytes);
    AL(p->ctx_v[s], ctx_bytes);
  }
  AL(p->ctx_state, (size_t)Bm * 2 * sizeof(int));   // per robot {active slot, prefix length}
  // conditioning rows: the time rows (H, or B*H with a schedule per robot),
  // then the robots' offset rows
  const size_t rows_t = c.per_robot_times ? (size_t)Bm * H : (size_t)H;
  const size_t rows_c = rows_t + Bm, rows_a = (size_t)Bm * H, rows_y = (size_t)Bm * (H + F);
  AL(p->E, rows_c * D * es); AL(p->H1, rows_c * D * es); AL(p->HC, rows_c * D * es);
  AL(p->omega, (size_t)(D / 2) * sizeof(double));
  AL(p->modv, (rows_c + kCondCache) * p->mod_dim * 4);
  AL(p->cond, sizeof(CondCache));
  AL(p->cond_tkey, (size_t)H * sizeof(float));
  AL(p->cond_drow, (size_t)Bm * sizeof(int));
  AL(p->cond_commit, (size_t)2 * Bm * sizeof(int));
  AL(p->x, rows_a * D * 4);
  AL(p->Y, rows_y * D * es);
  AL(p->QKV, rows_y * p->nqkv * es);
  AL(p->O, rows_a * p->qdim * es);
  AL(p->GU, rows_a * 2 * Fm * 4);
  AL(p->Hm, rows_a * Fm * es);
  AL(p->V, rows_a * A * 4);
  p->attn_ws_bytes = (size_t)32 << 20;
  AL(p->attn_ws, p->attn_ws_bytes);
  p->tcws.ws_bytes = (size_t)24 << 20;
  p->tcws.n_counters = 4096;
  AL(p->tcws.ws, p->tcws.ws_bytes);
  AL(p->tcws.counters, p->tcws.n_counters * sizeof(int));
  AL(p->dn_times, rows_t * sizeof(float));
  AL(p->rel_mask, (size_t)A * sizeof(float));
  p->n_adapters = c.fop_adapter_every > 0 ? L / c.fop_adapter_every : 0;
  const int NA = p->n_adapters, nkv = 2 * c.n_kv_heads * c.head_dim;
  if (NA) {
    AL(p->a_wq, (size_t)NA * p->qdim * D * es);
    AL(p->a_wkv, (size_t)NA * nkv * D * es);
    AL(p->a_wo, (size_t)NA * D * p->qdim * es);
    AL(p->a_gamma, (size_t)NA * D * 4);
    AL(p->a_zgamma, (size_t)NA * D * 4);
    AL(p->a_gate, (size_t)NA * 4);
    AL(p->Ya, (size_t)Bm * H * D * es);
    AL(p->Za, (size_t)Bm * F * D * es);
    AL(p->Qa, (size_t)Bm * H * p->qdim * es);
    AL(p->KVa, (size_t)Bm * F * nkv * es);
    AL(p->XA, (size_t)Bm * H * p->qdim * es);
  }
  AL(p->seeds, Bm * sizeof(uint64_t));
  AL(p->counters, Bm * sizeof(uint64_t));
  AL(p->head_cnt, Bm * sizeof(int));
  AL(p->err, sizeof(int));
#undef AL
  p->tcws.err = p->err;
  if (e == cudaSuccess) {
    int dev = 0;
    e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&p->num_sms, cudaDevAttrMultiProcessorCount, dev);
  }
  if (e == cudaSuccess && p->dt == DT_BF16) {
    e = init_tc_gemm();
    p->use_tc = (e == cudaSuccess);
    if (e == cudaSuccess) e = init_attention_tc();
    p->use_tc_attn = (e == cudaSuccess) && attention_tc_supported(c.head_dim, c.n_q_heads / c.n_kv_heads);
  }
  if (e != cudaSuccess) {
    *errs = std::string("allocation: ") + cudaGetErrorString(e);
    plan_destroy(p);
    return e == cudaErrorMemoryAllocation ? RAVEL_ENOMEM : RAVEL_ECUDA;
  }

  // staging for host weights: the largest single tensor slice packed at once
  size_t stage = (size_t)D * p->mod_dim;
  stage = std::max(stage, (size_t)D * p->nqkv);
  stage = std::max(stage, (size_t)p->qdim * D);
  stage = std::max(stage, (size_t)D * Fm);
  float* staging = nullptr;
  if (!w.on_device) {
    e = cudaMalloc((void**)&staging, stage * sizeof(float));
    if (e != cudaSuccess) {
      *errs = "weight staging allocation failed";
      plan_destroy(p);
      return RAVEL_ENOMEM;
    }
  }
  {
    // embedding frequencies w_i = 2 pi / p_i, periods geometric from 4e-3 (i = 0) to 4 (i = D/2 - 1)
    std::vector<double> om(D / 2);
    for (int i = 0; i < D / 2; ++i) om[i] = 6.283185307179586 / (4e-3 * std::pow(1000.0, (double)i / (double)(D / 2 - 1)));
    e = cudaMemcpy(p->omega, om.data(), om.size() * sizeof(double), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
      *errs = "embedding table upload failed";
      if (staging) cudaFree(staging);
      plan_destroy(p);
      return RAVEL_ECUDA;
    }
  }
  Packer pk{p, wp, staging};
  pk.transpose(w.t_w1, D, D, p->t_w1);
  pk.transpose(w.t_w2, D, D, p->t_w2);
  pk.transpose(w.d_w1, D, D, p->d_w1);
  pk.transpose(w.d_w2, D, D, p->d_w2);
  pk.transpose(w.mod_w, D, p->mod_dim, p->mod_w);
  for (int l = 0; l < L; ++l) {
    pk.transpose(w.w_qkv + (size_t)l * D * p->nqkv, D, p->nqkv, (char*)p->w_qkv + (size_t)l * p->nqkv * D * es);
    pk.transpose(w.w_o + (size_t)l * p->qdim * D, p->qdim, D, (char*)p->w_o + (size_t)l * D * p->qdim * es);
    char* gu = (char*)p->w_gu + (size_t)l * 2 * Fm * D * es;
    pk.transpose(w.w_gate + (size_t)l * D * Fm, D, Fm, gu, 1, 0);
    pk.transpose(w.w_up + (size_t)l * D * Fm, D, Fm, gu, 1, 64);
    pk.transpose(w.w_down + (size_t)l * Fm * D, Fm, D, (char*)p->w_down + (size_t)l * D * Fm * es);
  }
  pk.transpose(w.out_w, D, A, p->out_w);
  for (int i = 0; i < NA; ++i) {
    const int nkv2 = 2 * c.n_kv_heads * c.head_dim;
    pk.transpose(w.a_wq + (size_t)i * D * p->qdim, D, p->qdim, (char*)p->a_wq + (size_t)i * p->qdim * D * es);
    pk.transpose(w.a_wkv + (size_t)i * D * nkv2, D, nkv2, (char*)p->a_wkv + (size_t)i * nkv2 * D * es);
    pk.transpose(w.a_wo + (size_t)i * p->qdim * D, p->qdim, D, (char*)p->a_wo + (size_t)i * D * p->qdim * es);
  }
  if (NA) {
    pk.copy_f32(w.a_gamma, (size_t)NA * D, p->a_gamma);
    pk.copy_f32(w.a_zgamma, (size_t)NA * D, p->a_zgamma);
    pk.copy_f32(w.a_gate, (size_t)NA, p->a_gate);
  }
  pk.copy_f32(w.t_b1, D, p->t_b1);
  pk.copy_f32(w.t_b2, D, p->t_b2);
  pk.copy_f32(w.d_b1, D, p->d_b1);
  pk.copy_f32(w.d_b2, D, p->d_b2);
  pk.copy_f32(w.mod_b, p->mod_dim, p->mod_b);
  pk.copy_f32(w.in_w, (size_t)A * D, p->in_w);
  pk.copy_f32(w.in_b, D, p->in_b);
  pk.copy_f32(w.fop_gamma, (size_t)L * D, p->fop_gamma);
  pk.copy_f32(w.out_b, A, p->out_b);
  if (pk.err == cudaSuccess) pk.err = cudaDeviceSynchronize();
  if (staging) cudaFree(staging);
  if (pk.err != cudaSuccess) {
    *errs = std::string("weight packing: ") + cudaGetErrorString(pk.err);
    plan_destroy(p);
    return RAVEL_ECUDA;
  }
  return RAVEL_OK;
}

// ---------------------------------------------------------------------------- the step

cudaError_t run_gemm(const StepPlan& p, const GemmArgs& g, cudaStream_t st) {
  if (p.use_tc && tc_gemm_supported(g)) return launch_gemm_tc(g, p.tcws, p.num_sms, st);
  if (g.epi == EPI_GEGLU) return cudaErrorNotSupported;
  return launch_gemm_simt(g, p.dt, st);
}

int& enqueue_fail_kind() {
  static thread_local int k = -1;
  return k;
}

const char* kernel_kind_name(int k) {
  static const char* const names[KK_COUNT] = {"embed", "gemm_cond", "gemm_mod", "in_proj", "norm", "gemm_qkv",
                                              "attention", "gemm_o", "gemm_gate_up", "geglu", "gemm_down",
                                              "gemm_out", "tail", "cond_cache", "adapter", "head_tail",
                                              "launch_gap"};
  return (k >= 0 && k < KK_COUNT) ? names[k] : "unknown";
}

cudaError_t enqueue_step(const StepPlan& p, int B, const StepIO& io, cudaStream_t st, int* n_kernels,
                         LaunchTrace* trace, const DenoisePass* dn) {
  const ravel_config& c = p.cfg;
  const int D = c.width, L = c.layers, H = c.slots, A = c.action_dim, F = c.fop_tokens, Fm = c.mlp_dim;
  enqueue_fail_kind() = -1;
  const size_t es = p.esize;
  const Dtype dt = p.dt;
  int nk = 0;
  cudaError_t e = cudaSuccess;
  auto mark = [&](int kind) {
    if (!trace || e != cudaSuccess) return;
    cudaEvent_t ev;
    e = cudaEventCreate(&ev);
    if (e != cudaSuccess) return;
    trace->events.push_back(ev);
    trace->kinds.push_back(kind);
    e = cudaEventRecord(ev, st);
  };
#define RUN(kind, call)                 \
  do {                                  \
    if (e == cudaSuccess) {             \
      e = (call);                       \
      ++nk;                             \
      mark(kind);                       \
      if (e != cudaSuccess) enqueue_fail_kind() = (kind); \
    }                                   \
  } while (0)
  auto gemm = [&](const void* Aop, int lda, const void* W, int M, int N, int K, Epi epi, void* out, int ldo,
                  Dtype out_dt, const float* bias, int split_cap = 0, const int* skip = nullptr, int xbf16 = 0) {
    GemmArgs g{Aop, lda, W, K, M, N, K, epi, out, ldo, out_dt, bias};
    g.max_splits = split_cap;
    g.skip = skip;
    g.xbf16 = xbf16;
    return run_gemm(p, g, st);
  };
  auto rowp = [&](const void* base, size_t row, size_t ld) { return (const void*)((const char*)base + row * ld * es); };

  // conditioning: embeddings, the two MLPs, modulation (App. A.1)
  struct PdlScope {   // the step's kernels after the first may overlap their predecessors
    ~PdlScope() { pdl_enabled() = false; }
  } pdl_scope;
  // steady-state cache: in the paper's rolling schedule the slot times are
  // the same every step and the context age takes a handful of values, so
  // the modulation rows usually exist already; the launches below then
  // compute nothing (cond_check sets the skip flag)
  // time rows of the conditioning: the H slot times, or B*H with a schedule
  // per robot (norms then read robot b's row b*H + j: t_stride = H)
  const int Ht = c.per_robot_times ? B * H : H, t_stride = c.per_robot_times ? H : 0;
  CondArgs ca{p.cond, p.cond_tkey, p.cond_drow, p.cond_commit, io.slot_times, io.delta, Ht, B, c.max_batch,
              p.modv, p.mod_dim, (p.cond_cache && !c.per_robot_times) ? 1 : 0};
  const int* skip = &p.cond->skip;
  pdl_enabled() = false;
  RUN(KK_COND_CACHE, launch_cond_check(ca, st));
  pdl_enabled() = p.use_pdl && !trace;
  RUN(KK_EMBED, launch_embed(io.slot_times, Ht, io.delta, B, D, p.omega, p.E, dt, st, skip));
  RUN(KK_GEMM_COND, gemm(p.E, D, p.t_w1, Ht, D, D, EPI_STORE_SILU, p.H1, D, dt, p.t_b1, 0, skip));
  RUN(KK_GEMM_COND, gemm(rowp(p.E, Ht, D), D, p.d_w1, B, D, D, EPI_STORE_SILU, (void*)rowp(p.H1, Ht, D), D, dt, p.d_b1,
                         0, skip));
  RUN(KK_GEMM_COND, gemm(p.H1, D, p.t_w2, Ht, D, D, EPI_STORE, p.HC, D, dt, p.t_b2, 0, skip));
  RUN(KK_GEMM_COND, gemm(rowp(p.H1, Ht, D), D, p.d_w2, B, D, D, EPI_STORE, (void*)rowp(p.HC, Ht, D), D, dt, p.d_b2, 0,
                         skip));
  RUN(KK_GEMM_MOD, gemm(p.HC, D, p.mod_w, Ht + B, p.mod_dim, D, EPI_STORE, p.modv, p.mod_dim, DT_F32, nullptr, 0,
                        skip));
  RUN(KK_COND_CACHE, launch_cond_commit(ca, st));
  // residual stream
  // in-projection; with the fused norms, also the first layer's first norm
  const bool fuse_in = p.fuse_norm && p.dt == DT_BF16 && D <= 4096;
  if (fuse_in) {
    const int FF0 = (io.obs && !(p.n_adapters > 0)) ? F : 0;
    RowNorm rn0{p.modv, p.mod_dim, p.mod_b, 0, p.cond_drow, B, H, FF0 ? io.obs : nullptr, F, p.fop_gamma, p.Y,
                      H + FF0};
    rn0.t_stride = t_stride;
    RUN(KK_IN_PROJ, launch_in_proj_norm(io.buffer, A, D, p.in_w, p.in_b, p.x, io.state, p.rel_mask, io.slot_times,
                                        rn0, dt, st));
  } else {
    RUN(KK_IN_PROJ, launch_in_proj(io.buffer, B * H, A, D, p.in_w, p.in_b, p.x, st, io.state, p.rel_mask,
                                   io.slot_times, H, t_stride));
  }
  const bool adapters = p.n_adapters > 0 && io.obs;
  const int FF = (io.obs && !adapters) ? F : 0;   // FOP tokens as keys of the self-attention
  const int RPR = H + FF;              // normed / QKV rows per robot: H slots, then the FOP tokens
  const int BH = B * H, BY = B * RPR;
  for (int l = 0; l < L; ++l) {
    NormArgs n1{p.x, B, H, D, p.modv, p.mod_dim, p.mod_b, 4 * l * D, FF ? io.obs : nullptr, F,
                p.fop_gamma + (size_t)l * D, p.Y, RPR, p.cond_drow};
    n1.t_stride = t_stride;
    if (l > 0 || !fuse_in) RUN(KK_NORM, launch_ada_norm(n1, dt, st));
    const void* wqkv = (const char*)p.w_qkv + (size_t)l * p.nqkv * D * es;
    if (p.use_tc_attn) {
      // the tensor-core attention reads K and V straight from the QKV rows
      GemmArgs gq{p.Y, D, wqkv, D, BY, p.nqkv, D, EPI_STORE, p.QKV, p.nqkv, dt, nullptr};
      gq.max_splits = p.split_cap[0];
      gq.xbf16 = 1;
      RUN(KK_GEMM_QKV, run_gemm(p, gq, st));
      AttnTcArgs at{p.QKV, p.nqkv, {p.ctx_k[0], p.ctx_k[1]}, {p.ctx_v[0], p.ctx_v[1]}, L, l,
                    c.max_batch, c.max_prefix, p.ctx_state, B, H, FF, c.n_q_heads, c.n_kv_heads, c.head_dim,
                    c.mask_mode, p.O, p.qdim, p.attn_ws, p.attn_ws_bytes, p.err, p.num_sms};
      int launched = 0;
      at.n_launched = &launched;
      RUN(KK_ATTENTION, launch_attention_tc(at, st));
      nk += launched - 1;   // RUN counted one launch; a split attention adds its combine kernel
    } else {
      RUN(KK_GEMM_QKV, gemm(p.Y, D, wqkv, BY, p.nqkv, D, EPI_STORE, p.QKV, p.nqkv, dt, nullptr));
      AttnArgs at{p.QKV, p.nqkv, p.ctx_k[0], p.ctx_k[1], p.ctx_v[0], p.ctx_v[1], p.ctx_state, l, c.max_batch,
                  c.max_prefix, B, H, FF, c.n_q_heads, c.n_kv_heads, c.head_dim, c.mask_mode, p.O, p.qdim, p.err};
      RUN(KK_ATTENTION, launch_attention_simt(at, dt, st));
    }
    RUN(KK_GEMM_O, gemm(p.O, p.qdim, (const char*)p.w_o + (size_t)l * D * p.qdim * es, BH, D, p.qdim, EPI_ADD_F32, p.x,
                        D, DT_F32, nullptr, p.split_cap[1], nullptr, 1));
    if (adapters && (l + 1) % c.fop_adapter_every == 0) {
      // gated cross-attention adapter: the action rows attend to the FOP tokens
      const int ai = (l + 1) / c.fop_adapter_every - 1, nkv = 2 * c.n_kv_heads * c.head_dim;
      NormArgs na{p.x, B, H, D, nullptr, 0, nullptr, 0, nullptr, 0, nullptr, p.Ya, H};
      na.act_gain = p.a_gamma + (size_t)ai * D;
      RUN(KK_ADAPTER, launch_ada_norm(na, dt, st));
      NormArgs nz{p.x, B, 0, D, nullptr, 0, nullptr, 0, io.obs, F, p.a_zgamma + (size_t)ai * D, p.Za, F};
      RUN(KK_ADAPTER, launch_ada_norm(nz, dt, st));
      RUN(KK_ADAPTER, gemm(p.Ya, D, (const char*)p.a_wq + (size_t)ai * p.qdim * D * es, BH, p.qdim, D, EPI_STORE, p.Qa,
                           p.qdim, dt, nullptr));
      RUN(KK_ADAPTER, gemm(p.Za, D, (const char*)p.a_wkv + (size_t)ai * nkv * D * es, B * F, nkv, D, EPI_STORE, p.KVa,
                           nkv, dt, nullptr));
      RUN(KK_ADAPTER, launch_fop_xattn(p.Qa, p.KVa, p.XA, B, H, F, c.n_q_heads, c.n_kv_heads, c.head_dim,
                                       p.a_gate + ai, dt, st));
      RUN(KK_ADAPTER, gemm(p.XA, p.qdim, (const char*)p.a_wo + (size_t)ai * D * p.qdim * es, BH, D, p.qdim, EPI_ADD_F32,
                           p.x, D, DT_F32, nullptr));
    }
    NormArgs n2{p.x, B, H, D, p.modv, p.mod_dim, p.mod_b, 4 * l * D + 2 * D, nullptr, 0, nullptr, p.Y, H, p.cond_drow};
    n2.t_stride = t_stride;
    RUN(KK_NORM, launch_ada_norm(n2, dt, st));
    const void* wgu = (const char*)p.w_gu + (size_t)l * 2 * Fm * D * es;
    GemmArgs gu{p.Y, D, wgu, D, BH, 2 * Fm, D, EPI_GEGLU, p.Hm, Fm, dt, nullptr};
    gu.max_splits = p.split_cap[2];
    gu.xbf16 = 1;
    if (p.use_tc && tc_gemm_supported(gu)) {
      RUN(KK_GEMM_GATE_UP, launch_gemm_tc(gu, p.tcws, p.num_sms, st));   // GeGLU fused in the epilogue
    } else {
      RUN(KK_GEMM_GATE_UP, gemm(p.Y, D, wgu, BH, 2 * Fm, D, EPI_STORE, p.GU, 2 * Fm, DT_F32, nullptr));
      RUN(KK_GEGLU, launch_geglu(p.GU, BH, Fm, p.Hm, dt, st));
    }
    RUN(KK_GEMM_DOWN, gemm(p.Hm, Fm, (const char*)p.w_down + (size_t)l * D * Fm * es, BH, D, Fm, EPI_ADD_F32, p.x, D,
                           DT_F32, nullptr, p.split_cap[3], nullptr, 1));
  }
  if (!dn && dt == DT_BF16 && A <= 32 && D % 4 == 0) {
    // final norm, velocity head and tail in one launch, about eight CTAs per SM
    TailArgs ta{io.buffer, p.V, io.slot_times, io.released, io.velocity, p.seeds, p.counters, B, H, A, io.state,
                p.rel_mask};
    ta.t_stride = t_stride;
    const int rpc = std::max(1, (B * H + 8 * p.num_sms - 1) / (8 * p.num_sms));
    HeadArgs hd{p.x, D, p.modv, p.mod_dim, p.mod_b, 4 * L * D, p.cond_drow, p.out_w, p.out_b, p.V, p.head_cnt, rpc};
    hd.t_stride = t_stride;
    RUN(KK_HEAD_TAIL, launch_head_tail(hd, ta, st));
    if (n_kernels) *n_kernels = nk;
    return e;
  }
  NormArgs nf{p.x, B, H, D, p.modv, p.mod_dim, p.mod_b, 4 * L * D, nullptr, 0, nullptr, p.Y, H, p.cond_drow};
  nf.t_stride = t_stride;
  RUN(KK_NORM, launch_ada_norm(nf, dt, st));
  RUN(KK_GEMM_OUT, gemm(p.Y, D, p.out_w, BH, A, D, EPI_STORE, p.V, A, DT_F32, p.out_b));
  if (dn) {
    RUN(KK_TAIL, launch_denoise_tail(io.buffer, p.V, io.velocity, B, H, A, dn->t_now, dn->t_next, st));
  } else {
    TailArgs ta{io.buffer, p.V, io.slot_times, io.released, io.velocity, p.seeds, p.counters, B, H, A, io.state,
                p.rel_mask};
    ta.t_stride = t_stride;
    RUN(KK_TAIL, launch_tail(ta, st));
  }
#undef RUN
  if (n_kernels) *n_kernels = nk;
  return e;
}

}  // namespace ravel
