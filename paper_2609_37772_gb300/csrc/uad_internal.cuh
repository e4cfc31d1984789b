// Internal declarations shared by the library's translation units.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace uad {

constexpr int kMaxSteps = 64;              // = UAD_MAX_STEPS
constexpr int kFlagStride = kMaxSteps + 1;  // host flag slots per robot (steps 1..64)

enum DType { F32 = 0, BF16 = 1 };

// Programmatic dependent launch. Kernels of the step loop are launched so that the next kernel's
// CTAs may start while the previous kernel drains; every kernel calls pdl_trigger() once it has
// started and pdl_wait() before it reads anything a predecessor wrote or writes anything a
// predecessor reads (pdl_wait returns at once for a kernel launched without the attribute).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
bool pdl_enabled();   // UAD_PDL=0 turns it off (debugging)

template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                            Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

// GEMM epilogues (out[m][n] from acc = sum_k A[m][k] * Wt[n][k]).
enum Epi {
  EPI_STORE = 0,       // out = acc (+ bias) (+ add_rows[m % add_mod][n])
  EPI_BIAS_SILU = 1,   // out = silu(acc + bias)
  EPI_RESID_GATE = 2,  // CUDA cores: resid[m][n] += gate(m, n) * (acc + bias); gate = 1 without gate_tab
  EPI_GEGLU = 3,       // rows interleaved (2j = gate, 2j+1 = up): out[m][j] = gelu_tanh(g) * u
  EPI_BIAS_GELU = 4,   // out = gelu_tanh(acc + bias)
  EPI_PARTIAL = 6,     // tensor cores: K split s writes its fp32 tile to plane s of out [splits][M][N]
  EPI_QKV_TC = 5,      // q/k rows pair-interleaved per head: RoPE, then scatter q -> Q, k -> K cache,
                       // v -> Vt cache (tensor-core attention layouts, see attn_tc.cu)
};

// Where the QKV projection epilogue (EPI_QKV_TC) writes, and the RoPE table it uses.
struct QkvTcOut {
  __nv_bfloat16* q = nullptr;        // [B][Hkv][G*H][dh]
  __nv_bfloat16* kcache = nullptr;   // [B][L][Hkv][NK][dh]
  __nv_bfloat16* vtcache = nullptr;  // [B][L][Hkv][dh][NKp]
  const float* rope = nullptr;       // [H][dh/2][2] (cos, sin) at positions P + i, or null
  int H = 0, P = 0, NK = 0, NKp = 0, dh = 0, G = 1, Hkv = 1, L = 0, layer = 0, qd = 0, kvd = 0;
};

struct GemmArgs {
  const void* A = nullptr; int lda = 0; int a_dtype = F32;  // activations [M][K]
  const void* W = nullptr; int w_dtype = F32;               // weights [N][K], K contiguous
  int M = 0, N = 0, K = 0;
  int epi = EPI_STORE;
  void* out = nullptr; int ldo = 0; int out_dtype = F32;
  const float* bias = nullptr;                     // [N]
  const float* add_rows = nullptr; int add_mod = 1; // EPI_STORE: + add_rows[(m % add_mod) * N + n]
  float* resid = nullptr; int ldr = 0;             // EPI_RESID_GATE target, fp32
  const float* gate_tab = nullptr; int gate_stride = 0;  // gate(m, n) = gate_tab[tau_row[m] * gate_stride + n]
  const int* tau_row = nullptr;
  QkvTcOut qkv;                                    // EPI_QKV_TC
  int n_store = 0;                                 // > 0: outputs n >= n_store are padding, not stored
};

struct NormArgs {
  float* h = nullptr; int ldh = 0;         // fp32 [M][W]
  // pending residual update applied first (resid_norm): h += gate * (sum of n_part planes + bias)
  const float* part = nullptr; int n_part = 0;   // planes [n_part][M][W]
  const float* rgate_tab = nullptr; int rgate_off = 0;  // gate(m, c) = rgate_tab[tau_row[m] * stride + rgate_off + c]
  const float* rbias = nullptr;            // [W]
  int M = 0, W = 0;
  int layer_norm = 0;                      // 0: RMSNorm, 1: LayerNorm (no affine)
  const float* tab = nullptr; int stride = 0; int scale_off = 0, shift_off = 0;  // modulation
  const int* tau_row = nullptr;
  void* out = nullptr; int ldo = 0; int out_dtype = F32;
};

struct AttnArgs {
  int n_heads = 0, n_kv_heads = 0, head_dim = 0, H = 0, B = 0;
  const void* q = nullptr; int q_ld = 0;                 // q[(b*H + i) * q_ld + hq*dh + d]
  const void* kp = nullptr; const void* vp = nullptr;    // prefix segment
  int P = 0; long long kp_bstride = 0; int kp_ld = 0;    //   kp[b*kp_bstride + p*kp_ld + g*dh + d]
  const void* kc = nullptr; const void* vc = nullptr;    // chunk segment (may be null)
  int kc_ld = 0;                                         //   kc[(b*H + i) * kc_ld + g*dh + d]
  const float* rope_cs = nullptr;                        // [H][dh/2][2] (cos, sin) at positions P+i
  void* out = nullptr; int out_ld = 0;                   // out[(b*H + i) * out_ld + hq*dh + d]
  int dtype = F32;
  float scale = 1.f;
  // few-query attention split over key chunks: partial rows and per-(robot, head, query block)
  // arrival counts (zero between launches: the last CTA of a group resets its count)
  float* split_ws = nullptr;
  unsigned* split_ctr = nullptr;
};
// Workspace of the few-query attention split over key chunks, in floats and counters.
size_t attn_few_ws_floats(int B, int n_heads, int H, int n_keys);
size_t attn_few_ctr_count(int B, int n_heads, int H);

// Per-step, per-token plan entry (built on the host).
enum PlanFlag { PF_ACTIVE = 1, PF_GHOST = 2, PF_RELEASE = 4, PF_EARLY = 8, PF_FROZEN = 16,
                PF_NEXT_X = 32, PF_NEXT_G = 64, PF_NEXT_REL = 128, PF_LAST = 256 };

struct PlanTok {
  int flags;
  float dx;       // 1/N_i (fp32) when active
};

struct EulerArgs {
  int B = 0, H = 0, D = 0, k = 0;
  const PlanTok* plan = nullptr;     // this step's [B][H]
  const float* gstep = nullptr;      // [B] fp32(1/N*_b)
  const int* last_step = nullptr;    // [B] N*_b
  const int* tail_count = nullptr;   // [B] executable tail size (0: no GAC)
  const unsigned char* gac_mask = nullptr;  // [D]
  const int* tail_flag = nullptr;    // [B][H] 1 if corrected by GAC
  const float* v = nullptr;          // [B*H][D]
  float* x = nullptr; float* g = nullptr; float* u = nullptr; float* rel = nullptr;
  float* final_out = nullptr; float* ghost_out = nullptr; float* E_out = nullptr;  // device
  float* host_rel = nullptr;         // mapped pinned [B][H][D]
  int* host_flags = nullptr;         // mapped pinned [B][UAD_MAX_STEPS + 1]
  const int* epoch = nullptr;        // device scalar
  const int* rot_dim = nullptr;      // device scalar: first rotation-vector dimension, -1 none
  int* nonfinite = nullptr;
  int* evals = nullptr;                  // velocity evaluations consumed this chunk
  unsigned long long* stamps = nullptr;  // [UAD_MAX_STEPS + 1], [0] = start
};

// kernels_simt.cu
constexpr int kGemvMaxK = 8192;
void launch_gemm_simt(const GemmArgs& a, cudaStream_t s);
bool gemv_rows_ok(const GemmArgs& a);                     // tiny-side projection (N or K <= 64)
void launch_gemv_rows(const GemmArgs& a, cudaStream_t s);
void launch_norm(const NormArgs& a, cudaStream_t s);   // applies the pending residual if part != null
void launch_attention(const AttnArgs& a, cudaStream_t s);
void launch_euler(const EulerArgs& a, cudaStream_t s);
void launch_euler_prepare();   // shared memory for H x D GAC terms (up to 256 x 64)
void launch_begin(const float* noise, float* x, float* g, float* u, int n, int* nonfinite, int* evals,
                  unsigned long long* stamps, cudaStream_t s);
// dst[(n * mult + off) * K + k] = src[k * N + n]: transpose [K][N] -> rows of K, convert dtype
void launch_relayout(const float* src, int K, int N, void* dst, int dtype, int mult, long long off,
                     cudaStream_t s);
size_t attention_smem_bytes(int dh);
void launch_attention_prepare(int dh);  // opt in to > 48 KB dynamic shared memory (call once)
void launch_convert(const void* src, int src_dtype, void* dst, int dst_dtype, long long n, cudaStream_t s);
void launch_so3_check(const float* w, int n, float* log_exp, float* log_comp, cudaStream_t s);
// y[m][n] = SiLU(x[m][n] + tab[tau_row[m] * stride + off + n]) in dtype dt (the input MLP of the
// time-concatenating expert: the table holds e(tau) W_it + b_it per flow time)
void launch_add_tau_silu(const float* x, const float* tab, int stride, int off, const int* tau_row, int M, int N,
                         void* y, int dt, cudaStream_t s);

// gemm_tc.cu: tcgen05 projection GEMM (bf16 operands, fp32 accumulation in TMEM)
constexpr int kTcMaxStages = 4;        // <= ~97 KB of shared memory: two CTAs fit one SM
struct TcGemmArgs {
  const void* w_tiled = nullptr;   // [N/128][K/64] blocks of 128 x 64 bf16, 128B-swizzled K-major
  int M = 0, N = 0, K = 0, splits = 1;
  int epi = EPI_STORE;
  void* out = nullptr; int ldo = 0; int out_dtype = BF16;
  const float* bias = nullptr;
  QkvTcOut qkv;                    // EPI_QKV_TC
  int n_store = 0;                 // EPI_STORE: > 0: rows n >= n_store are padding (not stored, no bias)
  float* acc = nullptr;            // split-K accumulator [M][N] fp32, zero between launches
  int* counters = nullptr;         // split-K arrival counters per output tile, zero between launches
  int* err = nullptr;              // set to a nonzero code if a bounded wait gave up
  int wide = 0;                    // 1: the persistent wide form (one CTA per SM walking units of
                                   // tn tokens x 128 weight rows x a K range), 0: narrow split-K tiles
  int tn = 0;                      // persistent form: tokens per tile (256, 192 or 128)
  unsigned long long* trace = nullptr;  // optional: 16 global-timer stamps per CTA (phase times)
};
size_t gemm_tc_smem_bytes(int stages, int epi, int M);
// 2-D TMA descriptor of a bf16 activation matrix [rows][K] (64 x 64 boxes, 128-byte swizzle,
// zero fill past the last row). 0 on success.
int encode_act_tmap(CUtensorMap* m, const void* base, int K, int rows);
void gemm_tc_prepare();
int gemm_tc_splits(int M, int N, int K, int sms, int epi);
int gemm_tc_use_wide(int M, int N, int sms);    // 1: the persistent wide form serves this projection
// The tile plan of one projection (wide form, tokens per tile, K splits) into a.
void gemm_tc_plan(int M, int N, int K, int sms, int epi, TcGemmArgs* a);
void launch_gemm_tc(const CUtensorMap* tmx, const TcGemmArgs& a, cudaStream_t s);
// element (k, n) of src [K][N] -> row n' * mult + off, column k of the tiled bf16 layout (K cols),
// where n' = n, or with rope_dh > 0 the head-local pair interleave (d, d + dh/2) -> (2d, 2d + 1)
void launch_relayout_tiled(const float* src, int K, int N, void* dst, int mult, long long off, int rope_dh,
                           cudaStream_t s);

// attn_tc.cu: tensor-core attention over [prefix ; chunk] keys
struct AttnTcArgs {
  int batch = 0, n_layers = 0, layer = 0, n_kv_heads = 0, group = 1, head_dim = 0, H = 0, prefix = 0;
  int n_keys = 0, nk_pad = 0, rows = 0, r_pad = 0;
  float scale_log2 = 0.f;              // log2(e) / sqrt(dh)
  __nv_bfloat16* q = nullptr;          // [B][Hkv][rows][dh]
  __nv_bfloat16* kcache = nullptr;     // [B][L][Hkv][n_keys][dh]
  __nv_bfloat16* vtcache = nullptr;    // [B][L][Hkv][dh][nk_pad]
  float* part_o = nullptr;             // [B*Hkv][chunks][r_pad][dh]
  float* part_ml = nullptr;            // [B*Hkv][chunks][r_pad][2]
  __nv_bfloat16* out = nullptr; int out_ld = 0;   // o [B*H][Hq*dh]
  int* err = nullptr;
};
// k: 128-key boxes; k2: 64-key boxes (step kernel); vt: 64-key Vt boxes of all head dims; vt2: of
// half of them (the one-pass kernel's split form)
struct AttnTcMaps { CUtensorMap q, k, vt, k2, vt2; };
size_t attn_tc_smem_bytes(int dh);
int attn_tc_prepare(AttnTcMaps* maps, const AttnTcArgs& a, int batch_max);  // 0 on success
int attn_tc_chunks(int n_keys);
int attn_tc_max_keys();
int attn_tc_rpad(int rows);
// two kernels (split-KV attention, combine), or the one-pass kernel alone when
// attn_tc_use_two_pass (many query tiles)
void launch_attn_tc(const AttnTcMaps& maps, const AttnTcArgs& a, cudaStream_t s);
bool attn_tc_use_two_pass(const AttnTcArgs& a);
void launch_kv_prefix(const void* k, const void* v, int src_dtype, const AttnTcArgs& a, int robot, cudaStream_t s);

// ---- persistent evaluation kernel (adaRMS experts, bf16, few tokens) ----------------------
constexpr int kStepMaxRows = 64;      // tokens + distinct flow times per evaluation (MMA N side)
constexpr int kStepMaxShift = 16;     // distinct flow times per evaluation
constexpr int kStepMaxATiles = 8;     // weight tiles per CTA and projection
constexpr int kStepMaxRing = 12;      // weight ring slots of 16 KB
constexpr int kStepMaxChunks = 32;    // 64-key chunks per (robot, KV head)
constexpr int kStepMaxNB = 64;        // 128-row output blocks per projection
constexpr int kStepMaxQTiles = 64;    // (robot, KV head, 128-row query tile) triples per evaluation
constexpr int kStepBarriersPerLayer = 6;
constexpr int kStepMaxWidth = 2048;   // model width, a multiple of 512
// Per-launch synchronisation block (zeroed before every launch): grid-barrier counters,
// per-output-block arrival counters, row sums of squares of the residual stream, per-query-tile
// counts of finished attention chunks, per-layer counts of finished epilogue shares (qkv, o,
// gate/up) and chunk merges, and the count of CTAs that finished the final phase.
__host__ __device__ constexpr size_t step_sync_words(int L) {
  return (size_t)(1 + kStepBarriersPerLayer * L) + (size_t)L * 4 * kStepMaxNB + (size_t)(L + 1) * 2 * kStepMaxRows +
         (size_t)L * kStepMaxQTiles + (size_t)L * 4 + 1;
}
struct StepArgs {
  int M = 0, B = 0, H = 0, W = 0, F = 0, D = 0, L = 0;
  int qd = 0, kvd = 0, qkvd = 0, n_heads = 0, n_kv_heads = 0, group = 0, dh = 0;
  int P = 0, n_keys = 0, nk_pad = 0, rows = 0, r_pad = 0, n_chunks = 0;
  int ring = 0;                        // weight ring slots
  int rope = 0;                        // q/k rows pair-interleaved per head, rotated by rope_cs
  float scale_log2 = 0.f;              // log2(e) / sqrt(dh)
  const int* tau_row = nullptr;        // [M] modulation row of each token at this step
  const int* sidx = nullptr;           // [M] index of each token's flow time among the step's distinct ones
  const int* sinfo = nullptr;          // [1 + kStepMaxShift]: count of distinct flow times, their rows
  const float* tab = nullptr; int rowlen = 0;
  const float* u = nullptr;            // [M][D] model input
  const void* w_in = nullptr; const float* b_in = nullptr;     // bf16 [W][D]
  const void* w_out = nullptr; const float* b_out = nullptr;   // bf16 [D][W]
  float* v = nullptr;                  // [M][D] velocity
  float* h = nullptr;                  // [M][W] residual stream
  __nv_bfloat16* z = nullptr;          // [kStepMaxRows][W] projection input rows (see step_tc.cu)
  __nv_bfloat16* o = nullptr;          // [M][qd] attention output
  __nv_bfloat16* act = nullptr;        // [M][F] MLP activation
  float *acc_qkv = nullptr, *acc_o = nullptr, *acc_gu = nullptr, *acc_d = nullptr;  // zero between uses
  const void* const* wl = nullptr;     // [L][4] tiled weights: qkv, o, gate/up, down
  __nv_bfloat16 *q = nullptr, *kcache = nullptr, *vtcache = nullptr;   // tensor-core attention layouts
  __nv_bfloat16* part_o = nullptr;     // [B*Hkv][n_chunks][r_pad][dh] unnormalised partial O rows
  float* part_ml = nullptr;            // [B*Hkv][n_chunks][r_pad][2] (max, sum) of each partial row
  const float* rope_cs = nullptr;      // [H][dh/2][cos, sin]
  unsigned* sync = nullptr;            // step_sync_words(L) words, zeroed per launch
  int* err = nullptr;
  unsigned long long wait_ns = 2000000000ull;   // bound on any single wait
  unsigned unreachable = 0;            // testing aid: arrivals the first grid barrier waits for in excess
  EulerArgs eu;                        // the step epilogue, run by the last CTA to finish
};
struct StepMaps { CUtensorMap z, o, act, q, k, vt; };   // k: 64-key boxes
size_t step_smem_bytes(int dh, int ring);
int step_ring_slots(int dh, int smem_optin);           // ring slots that fit (may be < 3: unusable)
int step_prepare(int dh, int ring, int* blocks_per_sm); // 0 on success
// Tiles per CTA of the largest projection under the kernel's tile assignment (grid = `ctas`):
// every CTA's tiles of a projection lie in one 128-row output block. 0 if a projection has
// more output blocks than CTAs or than kStepMaxNB.
int step_max_tiles(int ctas, const int (*shapes)[2], int n);
int launch_step(const StepMaps& m, const StepArgs& a, int grid, cudaStream_t s);   // grid = SMs

}  // namespace uad
