// The step plan: every device buffer of one handle and the kernel sequence of
// one rolling step.
#pragma once

#include <cuda_runtime.h>

#include <string>
#include <vector>

#include "../../include/ravel.h"
#include "kernels.h"

namespace ravel {

// Caller-owned pointers of one ravel_roll_step call (captured into the graph).
struct StepIO {
  float* buffer;
  const float* slot_times;
  const void* obs;
  const float* delta;
  float* released;
  float* velocity;
  const float* state = nullptr;   // [B][A] latest robot state: absolute buffer, relative expert
};

struct StepPlan {
  ravel_config cfg{};
  Dtype dt = DT_F32;
  size_t esize = 4;
  int nqkv = 0, qdim = 0, mod_dim = 0;
  // packed weights, K-major [out][in] in dtype; biases / gains fp32
  void *t_w1 = nullptr, *t_w2 = nullptr, *d_w1 = nullptr, *d_w2 = nullptr, *mod_w = nullptr;
  void *w_qkv = nullptr, *w_o = nullptr, *w_gu = nullptr, *w_down = nullptr, *out_w = nullptr;
  float *t_b1 = nullptr, *t_b2 = nullptr, *d_b1 = nullptr, *d_b2 = nullptr, *mod_b = nullptr;
  float *in_w = nullptr, *in_b = nullptr, *fop_gamma = nullptr, *out_b = nullptr;
  // VLM context double buffer [2] x [L][Bmax][Hkv][Pmax][hd] (K and V alike) and its
  // device state per robot {active slot, prefix length}
  void* ctx_k[2] = {nullptr, nullptr};
  void* ctx_v[2] = {nullptr, nullptr};
  int* ctx_state = nullptr;
  // activations
  void* E = nullptr;      // [H+Bmax][D]  sinusoidal embeddings (times, then offsets)
  double* omega = nullptr;   // [D/2] angular frequencies of the embedding
  void* H1 = nullptr;     // [H+Bmax][D]  first MLP layer (SiLU)
  void* HC = nullptr;     // [H+Bmax][D]  MLP outputs h_t, h_delta
  float* modv = nullptr;  // [H+Bmax+kCondCache][mod_dim]  h @ W_mod (bias added in the norms):
                          // slot-time rows, this step's offset rows, cached offset rows
  CondCache* cond = nullptr;   // steady-state conditioning cache (kernels.h)
  float* cond_tkey = nullptr;  // [H]
  int* cond_drow = nullptr;    // [Bmax]
  int* head_cnt = nullptr;     // [Bmax] finished-row counters of the fused head kernel (zero between launches)
  int* cond_commit = nullptr;  // [2 Bmax]
  bool cond_cache = true;
  float* x = nullptr;     // [Bmax*H][D]  residual stream
  void* Y = nullptr;      // [Bmax*(H+F)][D]  normed rows (actions, then FOP tokens)
  void* QKV = nullptr;    // [Bmax*(H+F)][nqkv]
  void* O = nullptr;      // [Bmax*H][Hq*hd]
  float* GU = nullptr;    // [Bmax*H][2Fm]  interleaved gate/up (SIMT path)
  void* Hm = nullptr;     // [Bmax*H][Fm]
  float* V = nullptr;     // [Bmax*H][A]   velocity
  float* attn_ws = nullptr;  // split-KV partials of the tensor-core attention
  size_t attn_ws_bytes = 0;
  bool use_tc_attn = false;
  bool use_pdl = true;      // Programmatic Dependent Launch between the step's kernels
  // split-K caps of the layer GEMMs {QKV, O, gate/up, down} (0: from the shape)
  int split_cap[4] = {0, 0, 0, 0};
  TcWorkspace tcws{};       // split-K workspace of the tensor-core GEMM
  int num_sms = 0;
  bool use_tc = false;      // bf16 projections on tcgen05
  float* dn_times = nullptr;   // [H] flow times of a synchronous denoising pass (all equal)
  float* rel_mask = nullptr;   // [A] 1 = a dimension the expert predicts relative to the robot state
  bool fuse_norm = true;       // bf16: the in-projection also writes the first layer's first norm
  // FOP adapters (cfg.fop_adapter_every > 0): packed K-major weights, gains,
  // gates and their activations
  int n_adapters = 0;
  void *a_wq = nullptr, *a_wkv = nullptr, *a_wo = nullptr;
  float *a_gamma = nullptr, *a_zgamma = nullptr, *a_gate = nullptr;
  void *Ya = nullptr, *Za = nullptr, *Qa = nullptr, *KVa = nullptr, *XA = nullptr;
  uint64_t* seeds = nullptr;
  uint64_t* counters = nullptr;
  int* err = nullptr;
  std::vector<void*> allocs;
};

bool validate_config(const ravel_config& c, std::string* why);
ravel_status plan_create(StepPlan* p, const ravel_config& c, const ravel_weights& w, std::string* err);
void plan_destroy(StepPlan* p);

// Kernel kinds of one step (per-launch profiling labels).
enum KernelKind {
  KK_EMBED = 0, KK_GEMM_COND, KK_GEMM_MOD, KK_IN_PROJ, KK_NORM, KK_GEMM_QKV, KK_ATTENTION, KK_GEMM_O,
  KK_GEMM_GATE_UP, KK_GEGLU, KK_GEMM_DOWN, KK_GEMM_OUT, KK_TAIL, KK_COND_CACHE, KK_ADAPTER,
  KK_HEAD_TAIL,    // final norm + velocity head + tail in one launch (bf16)
  KK_LAUNCH_GAP,   // an empty kernel timed like the step's launches (ravel_profile_step)
  KK_COUNT
};
const char* kernel_kind_name(int k);
// The kernel kind whose launch failed last in enqueue_step on this thread (-1: none)
int& enqueue_fail_kind();

// Optional per-launch trace: an event recorded after every launch.
struct LaunchTrace {
  std::vector<cudaEvent_t> events;   // events[i] recorded after launch i
  std::vector<int> kinds;
};

// One projection GEMM through the step's dispatcher (tcgen05 for bf16 when
// the shapes allow, SIMT otherwise).
cudaError_t run_gemm(const StepPlan& p, const GemmArgs& g, cudaStream_t st);

// One pass of the full-horizon (synchronous) denoising: every slot at flow
// time t_now, Euler step t_now - t_next, no release / shift / append.
struct DenoisePass {
  float t_now, t_next;
};

// Enqueue one rolling step for `B` robots on `st` (no synchronisation, graph
// capture safe when trace == nullptr).  *n_kernels receives the number of
// kernel launches.  With `dn`, the same expert pass ends in the synchronous
// denoising update instead of the rolling tail.
cudaError_t enqueue_step(const StepPlan& p, int B, const StepIO& io, cudaStream_t st, int* n_kernels,
                         LaunchTrace* trace = nullptr, const DenoisePass* dn = nullptr);

}  // namespace ravel
