// Internal launch API of the rolling-step kernels (host side).  Every launcher
// enqueues on `st` and returns the launch's cudaError_t.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace ravel {

enum Dtype { DT_F32 = 0, DT_BF16 = 1 };

// Bits of the device error word (one int in HBM, OR-ed by kernels, read by the host).
enum : int {
  ERR_PREFIX_LEN = 1 << 0,   // the active context's prefix length was out of range
  ERR_TIMEOUT = 1 << 1,      // a bounded mbarrier / flag wait ran out
  ERR_SHAPE = 1 << 2,        // a kernel was launched with sizes it cannot handle
};

// Kernel attributes (dynamic shared memory limits); called once per handle,
// outside any stream capture.
cudaError_t init_simt_kernels();

// ---- weight packing ---------------------------------------------------------
// dst[n][k] = src[k][n] converted to `dt` (src float32 [K, N] row-major).
// interleave64: dst row of column n is (n/64)*128 + off + n%64 (gate/up tiles).
cudaError_t launch_pack_transpose(const float* src, int K, int N, void* dst, Dtype dt, int interleave64,
                                  int off, cudaStream_t st);
cudaError_t launch_convert(const float* src, size_t n, void* dst, Dtype dt, cudaStream_t st);

// ---- conditioning -------------------------------------------------------------
// Steady-state cache of the conditioning (the modulation rows of the H slot
// times, and of up to kCondCache distinct context offsets).  cond_check
// compares this step's slot times and offsets with the cached keys, maps each
// robot to the modv row of its offset part (drow), lists the rows to copy
// into the cache after the modulation GEMM, and sets `skip` when every row is
// cached (the conditioning launches then compute nothing); cond_commit copies
// the listed rows.  modv rows: [0, H) slot times, [H, H + Bmax) this step's
// offsets, [H + Bmax, H + Bmax + kCondCache) cached offsets.
constexpr int kCondCache = 16;
struct CondCache {
  int skip;                     // this step: every row cached
  int t_valid;                  // t_key holds the slot times of modv rows [0, H)
  int n_commit;
  int next;                     // round-robin victim
  int used[kCondCache];
  float delta[kCondCache];
};
struct CondArgs {
  CondCache* cc; float* t_key;  // [H]
  int* drow;                    // [Bmax] out: modv row of robot b's offset part
  int* commit;                  // [Bmax] pairs (src row, dst row) as 2 ints each -> [2 Bmax]
  const float* slot_times; const float* delta;
  int H, B, Bmax;
  float* modv; int mod_ld;
  int enabled;                  // 0: always compute, drow = H + b
};
cudaError_t launch_cond_check(const CondArgs& a, cudaStream_t st);
cudaError_t launch_cond_commit(const CondArgs& a, cudaStream_t st);
// E[r][:] = sinusoidal(x_r) for r < H (x = slot_times[r]) and H <= r < H+B
// (x = delta[r-H]); periods geometric from 4e-3 to 4; fp64 angles reduced mod 2 pi.
// omega: device fp64 [D/2] angular frequencies 2 pi / p_i.
cudaError_t launch_embed(const float* slot_times, int H, const float* delta, int B, int D, const double* omega,
                         void* E, Dtype dt, cudaStream_t st, const int* skip = nullptr);

// ---- generic projection GEMM: out[m][n] = sum_k A[m][k] W[n][k] (W K-major) ----
enum Epi { EPI_STORE = 0, EPI_STORE_SILU = 1, EPI_ADD_F32 = 2, EPI_GEGLU = 3 };

// adaRMSNorm of whole rows right after the in-projection (see NormArgs for
// the formula): action row (b, j) = residual row b*H + j, written to
// Y[b*row_pitch + j]; with fop, FOP row (b, f) written to Y[b*row_pitch + H + f].
struct RowNorm {
  const float* modv; int mod_ld; const float* mod_b; int off; const int* drow;
  int B, H;
  const void* fop; int F; const float* gamma;
  void* Y; int row_pitch;
  int t_stride = 0;   // as NormArgs (also the slot times' stride for the relative shift)
};
struct GemmArgs {
  const void* A; int lda;       // [M][K] activations of dtype dt
  const void* W; int ldw;       // [N][K] weights of dtype dt
  int M, N, K;
  Epi epi;
  void* out; int ldo;           // EPI_STORE*: dtype `out_dt`; EPI_ADD_F32: float, += result
  Dtype out_dt;
  const float* bias;            // [N] or null
  int max_splits = 0;           // tcgen05 path: cap on the split-K factor (0: chosen from the shape)
  const int* skip = nullptr;    // optional device flag: nonzero at run time -> the launch computes nothing
  // tcgen05 split-K inside a cluster: the splits' partials may travel between
  // the SMs in bf16 (half the bytes of fp32; the sum itself stays fp32), which
  // the step's projections take; 0 keeps them in fp32
  int xbf16 = 0;
};
cudaError_t launch_gemm_simt(const GemmArgs& g, Dtype dt, cudaStream_t st);

// tcgen05 / TMEM / TMA path (bf16 operands only).  EPI_GEGLU: W rows come in
// 128-row blocks of 64 gate rows then the 64 matching up rows; out is bf16
// [M][N/2] with out[m][f] = gelu_tanh(gate_f) * up_f.
struct TcWorkspace {
  float* ws; size_t ws_bytes;   // split-K partial tiles
  int* counters; int n_counters;   // per-tile arrival counters, zero between launches
  int* err;                     // device error word
};
cudaError_t init_tc_gemm();
bool tc_gemm_supported(const GemmArgs& g);
// cluster = true: split-K partials are reduced through distributed shared
// memory inside a thread-block cluster (no workspace); false: through the
// workspace `ws` with a last-arriving-CTA fix-up.
cudaError_t launch_gemm_tc(const GemmArgs& g, const TcWorkspace& ws, int num_sms, cudaStream_t st,
                           bool cluster = true);
// Fault injection for tests: the next `launches` tensor-core GEMM launches
// that run without a thread-block cluster make their MMA thread wait for an
// mbarrier arrival that nobody makes, with a 2 ms limit; each gives up,
// drains its copies, raises ERR_TIMEOUT and exits (no fault, no hang).
void debug_withhold_gemm(int launches);

// ---- adaRMSNorm rows ---------------------------------------------------------
// Action rows r < B*H (b = r / H, j = r % H):
//   Y[r] = x[r] * rsqrt(mean(x[r]^2) + 1e-6) * (1 + sc) + sh,
//   sc[c] = modv[j][off+c] + modv[H+b][off+c] + mod_b[off+c], sh likewise at off+D.
// FOP rows B*H + b*F + f (when fop != null): Y = z * rsqrt(mean(z^2)+1e-6) * (1 + gamma).
// Output row of action (b, j) is b*row_pitch + j, of FOP token (b, f) b*row_pitch + H + f.
struct NormArgs {
  const float* x; int B, H, D;
  const float* modv; int mod_ld; const float* mod_b; int off;
  const void* fop; int F; const float* gamma;
  void* Y; int row_pitch;
  const int* drow = nullptr;    // optional: row of modv holding robot b's offset part (default H + b)
  const float* act_gain = nullptr;   // optional [D]: action rows y = x rsqrt(mean(x^2)+eps) (1 + act_gain),
                                     // without modulation (the query rows of a FOP adapter)
  int t_stride = 0;             // modv time row of slot j of robot b: b * t_stride + j (H: a schedule per robot)
};
cudaError_t launch_ada_norm(const NormArgs& a, Dtype dt, cudaStream_t st);

// ---- action in-projection: x[b*H+j][c] = sum_a buf[b][j][a] in_w[a][c] + in_b[c] ----
// With `state` ([B][A], or null) the buffer holds absolute coordinates and
// the expert sees a - (1 - t_j) rel_mask * state_b (the relative ones).
cudaError_t launch_in_proj(const float* buf, int BH, int A, int D, const float* in_w, const float* in_b,
                           float* x, cudaStream_t st, const float* state = nullptr, const float* rel_mask = nullptr,
                           const float* slot_times = nullptr, int H = 1, int t_stride = 0);

// The in-projection (as launch_in_proj) of whole rows with the first layer's
// adaRMSNorm into rn.Y (action rows and, with rn.fop, FOP rows).
cudaError_t launch_in_proj_norm(const float* buf, int A, int D, const float* in_w, const float* in_b, float* x,
                                const float* state, const float* rel_mask, const float* slot_times, const RowNorm& rn,
                                Dtype dt, cudaStream_t st);

// An empty kernel (one thread): the launch overhead of a timed eager replay.
cudaError_t launch_noop(cudaStream_t st);

// ---- GeGLU on the interleaved gate/up GEMM output --------------------------------
cudaError_t launch_geglu(const float* GU, int M, int Fm, void* Hm, Dtype dt, cudaStream_t st);

// ---- attention ---------------------------------------------------------------
struct AttnArgs {
  const void* qkv; int ld_qkv;      // rows of robot b: b*(H+F) + [H action slots, F FOP tokens]
  const void* ctx_k0; const void* ctx_k1;   // the two context slots [L][Bmax][Hkv][Pmax][hd]
  const void* ctx_v0; const void* ctx_v1;
  const int* ctx_state;             // device: [0] active slot, [1] prefix length
  int layer, Bmax, Pmax;
  int B, H, F, Hq, Hkv, hd;
  int mask_mode;
  void* out; int ld_out;            // [B*H][Hq*hd]
  int* err;
};
cudaError_t launch_attention_simt(const AttnArgs& a, Dtype dt, cudaStream_t st);

// tcgen05 attention (bf16).  K and V as the step stores them: the context
// slots [L][Bmax][Hkv][Pmax][hd], the FOP/slot keys in the QKV rows.
struct AttnTcArgs {
  const void* qkv; int ld_qkv;
  const void* ctx_k[2]; const void* ctx_v[2];
  int layers, layer, Bmax, Pmax;
  const int* ctx_state;
  int B, H, F, Hq, Hkv, hd, mask_mode;
  void* out; int ld_out;
  float* ws; size_t ws_bytes;
  int* err; int num_sms;
  int* n_launched = nullptr;   // optional: incremented by the number of kernels launched (1 or 2)
};
cudaError_t init_attention_tc();
bool attention_tc_supported(int hd, int G);
cudaError_t launch_attention_tc(const AttnTcArgs& a, cudaStream_t st);

// ---- gated cross-attention of a FOP adapter ------------------------------------------
// out[b*H + j][h*hd + c] = tanh(gate[0]) * sum_f softmax_f(q . k_f / sqrt(hd)) v_f[c] over the
// F FOP tokens of robot b: q from Q [B*H][Hq*hd], k / v from KV [B*F][2*Hkv*hd] (K heads, then
// V heads), query head h reading KV head h / (Hq / Hkv).  F <= 64.
cudaError_t launch_fop_xattn(const void* Q, const void* KV, void* out, int B, int H, int F, int Hq, int Hkv, int hd,
                             const float* gate, Dtype dt, cudaStream_t st);

// ---- rolling tail: Euler, release, shift, append ------------------------------------
struct TailArgs {
  float* buffer;             // [B][H][A] in place
  const float* vel;          // [B*H][A]
  const float* slot_times;   // [H]
  float* released;           // [B][A]
  float* vel_out;            // optional copy of vel ([B][H][A])
  const uint64_t* seeds;     // [B]
  uint64_t* counters;        // [B], advanced by one
  int B, H, A;
  const float* state = nullptr;      // optional [B][A]: absolute buffer, relative expert (see launch_in_proj):
  const float* rel_mask = nullptr;   // [A]; a' = a + dt (v + rel_mask * state)
  int t_stride = 0;                  // slot time of robot b's slot j: slot_times[b * t_stride + j]
};
cudaError_t launch_tail(const TailArgs& a, cudaStream_t st);

// The final adaRMSNorm, the velocity head and the tail in one launch (bf16
// weights, A <= 32): rows_per_cta slots of one robot per CTA write v = the
// head of their normed rows into a.vel; the robot's last CTA runs the tail.
struct HeadArgs {
  const float* x; int D;                       // residual stream [B*H][D]
  const float* modv; int mod_ld; const float* mod_b; int off; const int* drow;   // as NormArgs
  const void* w; const float* b;               // W_out [A][D] bf16, b_out [A]
  float* v;                                    // [B*H][A] velocity (= a.vel)
  int* cnt;                                    // [B] zero-initialised counters
  int rows_per_cta;
  int t_stride = 0;                            // as NormArgs
};
cudaError_t launch_head_tail(const HeadArgs& h, const TailArgs& a, cudaStream_t st);

// Synchronous (full-horizon) denoising: buffer += (t_now - t_next) * vel for
// every slot (vel_out optional copy); times[0..H-1] = t; a fresh chunk
// buffer[b][j] = noise(seeds[b], counters[b] + j), counters[b] += H.
cudaError_t launch_denoise_tail(float* buffer, const float* vel, float* vel_out, int B, int H, int A, float t_now,
                                float t_next, cudaStream_t st);
cudaError_t launch_fill_times(float* times, int H, float t, cudaStream_t st);
cudaError_t launch_chunk_noise(float* buffer, const uint64_t* seeds, uint64_t* counters, int B, int H, int A,
                               cudaStream_t st);

// buffer[b][j] = noise(seeds[b], j) for j < H; counters[b] = H.
cudaError_t launch_reset(float* buffer, const uint64_t* seeds, uint64_t* counters, int B, int H, int A,
                         cudaStream_t st);

// Busy-wait on the device for `ns` nanoseconds (globaltimer), then return.
cudaError_t launch_delay(unsigned long long ns, cudaStream_t st);

// Per-robot context updates: robot[i] switches to slot[i] with prefix length
// len[i] (flip), or receives its new context rows in slot[i] (scatter).
constexpr int kCtxListMax = 256;
struct CtxList {
  int n;
  int robot[kCtxListMax];
  int slot[kCtxListMax];
  int len[kCtxListMax];
};
// ctx_state [Bmax][2] = {slot, prefix length} per robot
cudaError_t launch_flip(int* ctx_state, const CtxList& f, cudaStream_t st);
// src [L][src_n][Hkv][P] rows of row_bytes, list entry i at source position
// i0 + i -> dst_{f.slot[i]} [L][Bmax][Hkv][Pmax] rows of robot f.robot[i]
cudaError_t launch_ctx_scatter(const void* src, int src_n, int i0, void* dst0, void* dst1, int L, int Bmax, int Hkv,
                               int P, int Pmax, size_t row_bytes, const CtxList& f, cudaStream_t st);

}  // namespace ravel
