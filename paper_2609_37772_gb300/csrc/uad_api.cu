// C ABI of the UAD library: context, weight layout, urgency plan, time-conditioning table,
// CUDA-graph step loop on a worker stream, pinned release hand-off, bounded waits.
#include <algorithm>
#include <chrono>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <numeric>
#include <string>
#include <thread>
#include <tuple>
#include <vector>

#include "../../include/uad.h"
#include "uad_internal.cuh"

using namespace uad;

namespace {

// A projection weight Wt [N][K] in the library layout: row-major (CUDA-core GEMM) or, for
// bf16 operands with N % 128 == 0 and K % 64 == 0, 128 x 64 swizzled blocks (tensor cores).
struct Lin {
  void* w = nullptr;
  bool tiled = false;
  int N = 0, K = 0;
};

struct LayerW {
  Lin wqkv;              // [(Hq + 2 Hkv) dh][W]: q rows, then k, then v
  Lin wo;                // [W][Hq dh]
  Lin wgu;               // ADARMS [2F][W], rows interleaved gate_j, up_j
  Lin wd;                // ADARMS [W][F]
  Lin wqc;               // DiT [Hq dh][W]
  Lin woc;               // DiT [W][Hq dh]
  void* wkc = nullptr;   // DiT [Hq dh][Pw] (used once per observation)
  void* wvc = nullptr;   // DiT [Hq dh][Pw]
  Lin w1;                // DiT [F][W]
  Lin w2;                // DiT [W][F]
  float* b1 = nullptr;   // DiT [F]
  float* b2 = nullptr;   // DiT [W]
};

struct Tensor {
  std::string name;
  long long rows, cols;  // blob layout [rows][cols] ([in][out] for linear weights)
  size_t off;            // float offset in the blob
};

}  // namespace

struct uad_ctx {
  uad_arch a{};
  int dev = 0, sms = 0;
  int es = 4;                 // bytes per weight / operand element
  int qd = 0, kvd = 0, qkvd = 0;  // Hq dh, Hkv dh, q+k+v width
  int rowlen = 0;             // floats per time-conditioning row: L * 6W + 2W
  int mmax = 0;               // max_batch * H
  std::string err;
  std::vector<void*> allocs;
  bool use_graphs = true;
  bool force_simt = false;     // UAD_GEMM=simt: CUDA-core GEMMs only (debugging)

  // tensor-core GEMM: TMA descriptors of the activation buffers, split-K workspace
  std::map<const void*, CUtensorMap> tmaps;
  // tensor-core attention (bf16 joint-attention experts): query matrix, K and Vt caches
  bool attn_tc = false;
  AttnTcArgs at0;                 // shapes and buffers; batch / layer set per launch
  AttnTcMaps atmaps;
  float* tc_acc = nullptr;
  int* tc_counters = nullptr;
  int* dev_err = nullptr;
  float* part = nullptr;          // K-split partial planes of the residual projections
  // persistent evaluation kernel (adaRMS, bf16, B * H <= 64): one launch per step
  bool step_ok = false;
  bool step_off = false;          // UAD_STEP=0: per-operation kernels only
  unsigned long long wait_ns = 2000000000ull;   // bound on any wait inside the persistent kernel
  int test_unreachable = 0;       // testing aid: extra arrivals the first phase count waits for
  int step_bmax = 0;              // robots per launch
  bool step_failed = false;       // a wait of the persistent kernel ran out: per-operation kernels
  bool cur_step = false;          // the chunk in flight runs on the persistent kernel
  StepArgs st0;                   // shapes and buffers; M, B, tau_row set per launch
  StepMaps smaps;
  double step_bytes_w = 0, step_flops_w = 0;   // weight bytes / 2 x params per evaluation

  // weights (library layout)
  float *t_w1 = nullptr, *t_b1 = nullptr, *t_w2 = nullptr, *t_b2 = nullptr;  // t_w* are dtype
  void* w_in = nullptr; float* b_in = nullptr;   // [W][D]
  void* w_out = nullptr; float* b_out = nullptr; // [D][W]
  Lin w_out_tc;                                  // the same padded to 128 rows, tiled (tensor cores)
  void* w_mod = nullptr; float* b_mod = nullptr; // [rowlen][W], all layers' modulation + final
  // time-concatenating expert (UAD_KIND_CONCAT): input MLP; e(tau) W_it + b_it sits in the table
  void* w_it = nullptr; float* b_it = nullptr;   // [W][W] (table fill)
  Lin w_ia, w_io; float* b_io = nullptr;          // [W][W] projections of the input MLP
  std::vector<LayerW> L;

  // time conditioning
  int tab_cap = 0, tab_rows = 0;
  float* tab = nullptr;        // [cap][rowlen]
  float *temb = nullptr, *tc1 = nullptr, *tc2 = nullptr;  // [cap][W] fill scratch
  std::map<std::pair<int, int>, int> tau_row;

  // per-position tables
  float* rope_cs = nullptr;    // [H][dh/2][2]
  float* pos_code = nullptr;   // [H][W] (DiT)

  // prefix
  void *kpre = nullptr, *vpre = nullptr;  // ADARMS [B][L][P][Hkv dh]; DiT [B][L][P][Hq dh]
  float* few_ws = nullptr;                // few-query attention: partial rows of the key chunks
  unsigned* few_ctr = nullptr;            // and their arrival counts (zero between launches)
  std::vector<int> has_prefix;

  // activations / state
  float* h = nullptr;                       // [mmax][W]
  void *y = nullptr, *qkv = nullptr, *qc = nullptr, *o = nullptr, *act = nullptr;
  float *v = nullptr, *x = nullptr, *g = nullptr, *u = nullptr, *rel = nullptr;
  float *fin = nullptr, *ghost = nullptr, *E = nullptr, *noise = nullptr;
  int* nonfinite = nullptr;
  int* evals = nullptr;
  unsigned long long* stamps = nullptr;

  // the finished chunk's status words, copied back in one batch of asynchronous copies (pinned)
  struct ChunkStatus { int derr, nonfinite, evals, pad; unsigned long long stamps[kFlagStride]; };
  ChunkStatus* status_host = nullptr;

  // plan block (device) + pinned staging
  unsigned char* plan_dev = nullptr;
  unsigned char* plan_host = nullptr;
  size_t plan_bytes_cap = 0;

  // release hand-off (mapped pinned)
  float* host_rel = nullptr; float* host_rel_dev = nullptr;
  int* host_flags = nullptr; int* host_flags_dev = nullptr;

  // per-kernel profiling (uad_profile_chunk): events around every launch of one eager chunk
  struct ProfRec { const char* name; double bytes, flops; int ev0, ev1; };
  bool prof_on = false;
  std::vector<ProfRec> prof;
  std::vector<cudaEvent_t> prof_ev;
  int prof_next = 0;

  cudaStream_t worker = nullptr;
  cudaEvent_t ev_in = nullptr, ev_done = nullptr;
  std::map<std::tuple<int, int, int>, cudaGraphExec_t> graphs;   // (robots, N*, persistent kernel)

  // in-flight chunk
  bool in_flight = false;
  int epoch = 0;
  int cur_B = 0, cur_steps = 0;
  std::vector<int32_t> cur_budgets;
  std::vector<int> cur_nstar;
  std::vector<unsigned long long> last_stamps;
  int last_steps = 0;
};

namespace {

int fail(uad_ctx* c, int code, const char* fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    c->err = buf;
  }
  return code;
}

#define CK(call)                                                                          \
  do {                                                                                    \
    cudaError_t e_ = (call);                                                              \
    if (e_ != cudaSuccess)                                                                \
      return fail(c, UAD_ECUDA, "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_),  \
                  __FILE__, __LINE__);                                                    \
  } while (0)

int dalloc(uad_ctx* c, void** p, size_t bytes) {
  *p = nullptr;
  if (bytes == 0) bytes = 16;
  cudaError_t e = cudaMalloc(p, bytes);
  if (e != cudaSuccess) {
    *p = nullptr;
    return fail(c, UAD_ENOMEM, "cudaMalloc(%zu) failed: %s", bytes, cudaGetErrorString(e));
  }
  c->allocs.push_back(*p);
  e = cudaMemset(*p, 0, bytes);
  if (e != cudaSuccess) return fail(c, UAD_ECUDA, "cudaMemset failed: %s", cudaGetErrorString(e));
  return UAD_OK;
}

template <class T>
int dalloc_t(uad_ctx* c, T** p, size_t count, size_t elem = sizeof(T)) {
  void* q = nullptr;
  int r = dalloc(c, &q, count * elem);
  *p = static_cast<T*>(q);
  return r;
}

std::vector<Tensor> blob_layout(const uad_arch& a) {
  std::vector<Tensor> t;
  size_t off = 0;
  auto add = [&](const std::string& n, long long r, long long cl) {
    t.push_back({n, r, cl, off});
    off += (size_t)(r * cl);
  };
  const long long W = a.width, D = a.action_dim, F = a.mlp_dim;
  const long long q = (long long)a.n_heads * a.head_dim, kv = (long long)a.n_kv_heads * a.head_dim;
  if (a.kind == UAD_KIND_CONCAT) {
    add("in_w", D, W); add("in_b", 1, W);
    add("ti_wa", W, W); add("ti_wt", W, W); add("ti_b", 1, W); add("to_w", W, W); add("to_b", 1, W);
    for (int l = 0; l < a.n_layers; ++l) {
      const std::string p = "l" + std::to_string(l) + ".";
      add(p + "wq", W, q); add(p + "wk", W, kv); add(p + "wv", W, kv); add(p + "wo", q, W);
      add(p + "wg", W, F); add(p + "wu", W, F); add(p + "wd", F, W);
    }
    add("out_w", W, D); add("out_b", 1, D);
    return t;
  }
  add("t_w1", W, W); add("t_b1", 1, W); add("t_w2", W, W); add("t_b2", 1, W);
  add("in_w", D, W); add("in_b", 1, W);
  for (int l = 0; l < a.n_layers; ++l) {
    const std::string p = "l" + std::to_string(l) + ".";
    if (a.kind == UAD_KIND_ADARMS) {
      add(p + "mod1_w", W, 3 * W); add(p + "mod1_b", 1, 3 * W);
      add(p + "wq", W, q); add(p + "wk", W, kv); add(p + "wv", W, kv); add(p + "wo", q, W);
      add(p + "mod2_w", W, 3 * W); add(p + "mod2_b", 1, 3 * W);
      add(p + "wg", W, F); add(p + "wu", W, F); add(p + "wd", F, W);
    } else {
      const long long Pw = a.prefix_width;
      add(p + "mod_w", W, 6 * W); add(p + "mod_b", 1, 6 * W);
      add(p + "wq", W, q); add(p + "wk", W, q); add(p + "wv", W, q); add(p + "wo", q, W);
      add(p + "wqc", W, q); add(p + "wkc", Pw, q); add(p + "wvc", Pw, q); add(p + "woc", q, W);
      add(p + "w1", W, F); add(p + "b1", 1, F); add(p + "w2", F, W); add(p + "b2", 1, W);
    }
  }
  add("modf_w", W, 2 * W); add("modf_b", 1, 2 * W); add("out_w", W, D); add("out_b", 1, D);
  return t;
}

int validate_arch(const uad_arch& a, std::string& why) {
  auto bad = [&](const char* m) { why = m; return UAD_EINVAL; };
  if (a.kind != UAD_KIND_ADARMS && a.kind != UAD_KIND_DIT && a.kind != UAD_KIND_CONCAT) return bad("kind");
  if (a.dtype != UAD_DTYPE_F32 && a.dtype != UAD_DTYPE_BF16) return bad("dtype");
  if (a.n_layers < 0 || a.n_layers > 256) return bad("n_layers");
  if (a.width < 32 || a.width % 32 || a.width > 8192) return bad("width (multiple of 32, <= 8192)");
  if (a.n_heads < 1 || a.n_kv_heads < 1 || a.n_heads % a.n_kv_heads) return bad("heads");
  if (a.head_dim != 64 && a.head_dim != 128 && a.head_dim != 256) return bad("head_dim in {64,128,256}");
  if (a.mlp_dim < 1 || a.mlp_dim > 65536) return bad("mlp_dim");
  if (a.action_dim < 1 || a.action_dim > 64) return bad("action_dim in 1..64");
  if (a.chunk_len < 1 || a.chunk_len > 256) return bad("chunk_len in 1..256");
  if (a.prefix_len < 0 || a.prefix_len > 16384) return bad("prefix_len");
  if (a.max_batch < 1 || a.max_batch > 1024) return bad("max_batch");
  if (a.kind == UAD_KIND_DIT) {
    if (a.n_kv_heads != a.n_heads) return bad("DiT needs n_kv_heads == n_heads");
    if (a.prefix_width < 1) return bad("prefix_width");
    if (a.prefix_len < 1) return bad("DiT needs prefix tokens");
    if (a.rope) return bad("DiT uses a position code, not RoPE");
  }
  return UAD_OK;
}

// Sinusoidal code of value t over `width` dims: [sin(scale t f_j), cos(scale t f_j)],
// f_j = 10000^(-j / (width/2)). Computed in double on the host.
void sinusoid_row(double t, int width, double scale, float* out) {
  const int half = width / 2;
  for (int j = 0; j < half; ++j) {
    const double f = std::exp(-std::log(10000.0) * j / half);
    out[j] = (float)std::sin(scale * t * f);
    out[half + j] = (float)std::cos(scale * t * f);
  }
}

// Offset in a table row of the time half of the time-concatenating expert's input MLP.
int concat_off(const uad_ctx* c) { return c->a.n_layers * 6 * c->a.width + 2 * c->a.width; }

// Fill time-conditioning rows for new flow times (App. C.1): time MLP then every layer's
// modulation Linear, one GEMM each over all new times; for the time-concatenating expert also
// e(tau) W_it + b_it.
int fill_times(uad_ctx* c, const std::vector<std::pair<int, int>>& fr, cudaStream_t s) {
  if (fr.empty()) return UAD_OK;
  const int n = (int)fr.size(), W = c->a.width;
  if (c->tab_rows + n > c->tab_cap)
    return fail(c, UAD_EINVAL, "more than %d distinct flow times", c->tab_cap);
  std::vector<float> e((size_t)n * W);
  for (int r = 0; r < n; ++r) sinusoid_row((double)fr[r].first / fr[r].second, W, 1000.0, &e[(size_t)r * W]);
  CK(cudaMemcpyAsync(c->temb, e.data(), e.size() * 4, cudaMemcpyHostToDevice, s));
  GemmArgs g;
  g.A = c->temb; g.lda = W; g.a_dtype = F32; g.W = c->t_w1; g.w_dtype = c->a.dtype;
  g.M = n; g.N = W; g.K = W; g.epi = EPI_BIAS_SILU; g.out = c->tc1; g.ldo = W; g.bias = c->t_b1;
  launch_gemm_simt(g, s);
  g.A = c->tc1; g.W = c->t_w2; g.out = c->tc2; g.bias = c->t_b2;
  launch_gemm_simt(g, s);
  g.A = c->tc2; g.W = c->w_mod; g.N = c->rowlen; g.epi = EPI_STORE; g.bias = c->b_mod;
  g.out = c->tab + (size_t)c->tab_rows * c->rowlen; g.ldo = c->rowlen;
  launch_gemm_simt(g, s);
  if (c->a.kind == UAD_KIND_CONCAT) {
    // the time half of the input MLP: e(tau) W_it + b_it after the (constant) modulation
    GemmArgs t;
    t.A = c->temb; t.lda = W; t.a_dtype = F32; t.W = c->w_it; t.w_dtype = c->a.dtype;
    t.M = n; t.N = W; t.K = W; t.epi = EPI_STORE; t.bias = c->b_it;
    t.out = c->tab + (size_t)c->tab_rows * c->rowlen + concat_off(c); t.ldo = c->rowlen;
    launch_gemm_simt(t, s);
  }
  CK(cudaGetLastError());
  for (int r = 0; r < n; ++r) c->tau_row[fr[r]] = c->tab_rows + r;
  c->tab_rows += n;
  return UAD_OK;
}

std::pair<int, int> reduce(int num, int den) {
  const int g = std::gcd(num, den);
  return {num / g, den / g};
}

// Plan block layout for a call with n_steps steps and B robots (16-byte aligned sections).
struct PlanLayout {
  size_t plan, tau, sidx, sinfo, gstep, last, tailc, tailf, mask, epoch, rot, total;
};
PlanLayout plan_layout(int n_steps, int B, int H, int D) {
  auto al = [](size_t x) { return (x + 15) & ~(size_t)15; };
  PlanLayout L{};
  const size_t M = (size_t)B * H;
  size_t o = 0;
  L.plan = o; o = al(o + n_steps * M * sizeof(PlanTok));
  L.tau = o; o = al(o + n_steps * M * 4);
  L.sidx = o; o = al(o + n_steps * M * 4);                        // persistent kernel: token -> flow time
  L.sinfo = o; o = al(o + n_steps * (1 + kStepMaxShift) * 4);     // count, rows of distinct flow times
  L.gstep = o; o = al(o + B * 4);
  L.last = o; o = al(o + B * 4);
  L.tailc = o; o = al(o + B * 4);
  L.tailf = o; o = al(o + M * 4);
  L.mask = o; o = al(o + D);
  L.epoch = o; o = al(o + 4);
  L.rot = o; o = al(o + 4);
  L.total = o;
  return L;
}

// One step of the per-token plan for one robot (host).
void plan_token(int k, int n_i, int ns, bool tr, int* flags, std::pair<int, int>* tau) {
  int f = 0;
  const bool early = n_i < ns;
  if (k <= ns) {
    const bool active = k <= n_i;
    if (active) { f |= PF_ACTIVE; *tau = reduce(k - 1, n_i); }
    else if (tr) { f |= PF_GHOST; *tau = reduce(k - 1, ns); }
    else { f |= PF_FROZEN; *tau = {1, 1}; }
    if (early) f |= PF_EARLY;
    if (early && k == n_i) f |= PF_RELEASE;
    if (k == ns) f |= PF_LAST;
    if (k + 1 <= n_i || k + 1 > ns) f |= PF_NEXT_X;
    else if (tr) f |= PF_NEXT_G;
    else f |= PF_NEXT_REL;
  } else {
    f |= PF_NEXT_X;
    *tau = {0, 1};
  }
  *flags = f;
}

// Brackets one kernel launch with timing events when profiling is on.
struct Mark {
  uad_ctx* c;
  cudaStream_t s;
  Mark(uad_ctx* c_, cudaStream_t s_, const char* name, double bytes, double flops) : c(c_), s(s_) {
    if (!c->prof_on) return;
    while ((int)c->prof_ev.size() < c->prof_next + 2) {
      cudaEvent_t e;
      cudaEventCreate(&e);
      c->prof_ev.push_back(e);
    }
    c->prof.push_back({name, bytes, flops, c->prof_next, c->prof_next + 1});
    cudaEventRecordWithFlags(c->prof_ev[c->prof_next], s, cudaEventRecordExternal);
    c->prof_next += 2;
  }
  ~Mark() {
    if (c->prof_on) cudaEventRecordWithFlags(c->prof_ev[c->prof.back().ev1], s, cudaEventRecordExternal);
  }
};

// Partial planes a residual projection [M][W] x [W][K]^T writes on the tensor cores.
size_t residual_planes(const uad_ctx* c, int M, int K) {
  TcGemmArgs t;
  gemm_tc_plan(M, c->a.width, K, c->sms, EPI_PARTIAL, &t);
  return (size_t)t.splits;
}

// Algorithmic HBM bytes of one projection: weights + activations in + output (+ residual r/w).
double gemm_bytes(const GemmArgs& g, int wes) {
  const double aes = g.a_dtype == BF16 ? 2 : 4, oes = g.out_dtype == BF16 ? 2 : 4;
  double b = (double)g.N * g.K * wes + (double)g.M * g.K * aes;
  if (g.epi == EPI_RESID_GATE) b += 8.0 * g.M * g.N;
  else if (g.epi == EPI_PARTIAL) b += 4.0 * g.M * g.N;
  else if (g.epi == EPI_GEGLU) b += oes * g.M * (g.N / 2);
  else b += oes * (double)g.M * g.N;
  return b;
}

// out = epi(A Wt^T): tensor cores when the weight is tiled, CUDA cores otherwise.
void gemm(uad_ctx* c, const Lin& w, GemmArgs g, cudaStream_t s) {
  g.W = w.w;
  if (!w.tiled) {
    // row-at-a-time kernel for a long K (action out) or few rows; a short K over many rows (the
    // action-in projection of a batch) goes to the tiled kernel, which reuses each weight tile
    // over 64 rows
    if (gemv_rows_ok(g) && (g.K > 64 || g.M <= 64)) launch_gemv_rows(g, s);
    else launch_gemm_simt(g, s);
    return;
  }
  TcGemmArgs t;
  t.w_tiled = w.w; t.M = g.M; t.N = g.N; t.K = g.K;
  gemm_tc_plan(g.M, g.N, g.K, c->sms, g.epi, &t);
  t.epi = g.epi; t.out = g.out; t.ldo = g.ldo; t.out_dtype = g.out_dtype; t.bias = g.bias;
  t.qkv = g.qkv; t.n_store = g.n_store; t.acc = c->tc_acc; t.counters = c->tc_counters; t.err = c->dev_err;
  launch_gemm_tc(&c->tmaps.at(g.A), t, s);
}

void gemm(uad_ctx* c, const void* w, GemmArgs g, cudaStream_t s) {
  Lin l;
  l.w = const_cast<void*>(w);
  gemm(c, l, g, s);
}

// Residual update h += gate(tau) * (A W^T + bias) (gate 1 without a table). Tensor-core
// weights: the K splits write fp32 partial planes and the update is left pending in `pend`
// for the next norm, which sums the planes in a fixed order, applies it and normalises in one
// pass over the row. CUDA-core weights: applied in the GEMM epilogue.
struct PendingResid {
  const float* part = nullptr; int n_part = 0;
  const float* gate_tab = nullptr; int gate_off = 0;
  const float* bias = nullptr;
};

void resid_gemm(uad_ctx* c, const Lin& w, GemmArgs g, int gate_off, const float* bias, PendingResid* pend,
                const char* name, cudaStream_t s) {
  const double flops = 2.0 * g.M * g.N * g.K;
  if (w.tiled) {
    g.epi = EPI_PARTIAL; g.out = c->part; g.ldo = g.N; g.out_dtype = F32;
    pend->part = c->part;
    pend->n_part = (int)residual_planes(c, g.M, g.K);
    pend->gate_tab = gate_off >= 0 ? c->tab : nullptr;
    pend->gate_off = gate_off;
    pend->bias = bias;
    Mark mk(c, s, name, gemm_bytes(g, c->es), flops);
    gemm(c, w, g, s);
    return;
  }
  g.epi = EPI_RESID_GATE; g.resid = c->h; g.ldr = g.N; g.bias = bias;
  if (gate_off >= 0) { g.gate_tab = c->tab + gate_off; g.gate_stride = c->rowlen; }
  Mark mk(c, s, name, gemm_bytes(g, c->es), flops);
  gemm(c, w, g, s);
}

// Norm of the residual stream, applying (and clearing) a pending residual update first.
void norm_after(uad_ctx* c, NormArgs n, PendingResid* pend, cudaStream_t s) {
  double by = (4.0 + c->es) * n.M * n.W;
  if (pend->part) {
    n.part = pend->part; n.n_part = pend->n_part;
    n.rgate_tab = pend->gate_tab; n.rgate_off = pend->gate_off; n.rbias = pend->bias;
    by += 8.0 * n.M * n.W;                     // partial sum in, residual row out
    *pend = PendingResid();
  }
  Mark mk(c, s, n.part ? "resid_norm" : "norm", by, 0);
  launch_norm(n, s);
}

// 2-D TMA descriptor of a bf16 activation buffer [rows][K]: 64 x 64 boxes, 128-byte swizzle,
// zero fill outside the buffer.
int make_tmap(uad_ctx* c, const void* base, int K, int rows) {
  CUtensorMap m;
  const int r = encode_act_tmap(&m, base, K, rows);
  if (r) return fail(c, UAD_ECUDA, "TMA descriptor encoding failed (%d)", r);
  c->tmaps[base] = m;
  return UAD_OK;
}

// The persistent evaluation kernel serves adaRMS experts with tensor-core attention when a
// chunk has at most 64 tokens per launch and the work fits its shared-memory plan; otherwise
// (and with UAD_STEP=0) every evaluation runs as per-operation kernels.
const char* step_unfit(uad_ctx* c, int* ring) {
  const uad_arch& a = c->a;
  const int W = a.width, F = a.mlp_dim, dh = a.head_dim;
  if (c->step_off) return "switched off";
  if (!c->attn_tc || a.kind != UAD_KIND_ADARMS) return "not an adaRMS expert with tensor-core attention";
  if (a.chunk_len > kStepMaxRows) return "chunk longer than 64 tokens";
  if (W % 512 || W > kStepMaxWidth) return "width";
  if (a.action_dim % 8) return "action dim";
  if (dh != 64 && dh != 128 && dh != 256) return "head dim";
  if ((c->at0.n_keys + 63) / 64 > kStepMaxChunks) return "too many keys";
  const int bmax = std::min(a.max_batch, kStepMaxRows / a.chunk_len);
  if (bmax * a.n_kv_heads * (c->at0.r_pad / 128) > kStepMaxQTiles) return "too many query tiles";
  const int shapes[4][2] = {{c->qkvd, W}, {W, c->qd}, {2 * F, W}, {W, F}};
  for (auto& sh : shapes)
    if (sh[0] % 128 || sh[1] % 64) return "projection shape";
  const int most = step_max_tiles(c->sms, shapes, 4);
  if (most < 1 || most > kStepMaxATiles) return "projection too large";
  for (const LayerW& w : c->L)
    if (!w.wqkv.tiled || !w.wo.tiled || !w.wgu.tiled || !w.wd.tiled) return "untiled weights";
  int optin = 0;
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, c->dev);
  *ring = step_ring_slots(dh, optin);
  if (*ring < 3) return "shared memory";
  // exactly one CTA per SM, all resident together (the grid barriers rely on it)
  int per_sm = 0;
  if (step_prepare(dh, *ring, &per_sm) || per_sm != 1) return "occupancy";
  return nullptr;
}

int step_setup(uad_ctx* c) {
  const uad_arch& a = c->a;
  int ring = 0;
  if (step_unfit(c, &ring)) return UAD_OK;
  const int H = a.chunk_len, W = a.width, F = a.mlp_dim, L = a.n_layers;
  const AttnTcArgs& t = c->at0;
  StepArgs& p = c->st0;
  c->step_bmax = std::min(a.max_batch, kStepMaxRows / H);
  p.H = H; p.W = W; p.F = F; p.D = a.action_dim; p.L = L;
  p.qd = c->qd; p.kvd = c->kvd; p.qkvd = c->qkvd; p.n_heads = a.n_heads; p.n_kv_heads = a.n_kv_heads;
  p.group = t.group; p.dh = a.head_dim; p.P = a.prefix_len; p.n_keys = t.n_keys; p.nk_pad = t.nk_pad;
  p.rows = t.rows; p.r_pad = t.r_pad; p.n_chunks = (t.n_keys + 63) / 64;
  p.ring = ring; p.rope = a.rope ? 1 : 0; p.scale_log2 = t.scale_log2;
  p.tab = c->tab; p.rowlen = c->rowlen; p.u = c->u;
  p.w_in = c->w_in; p.b_in = c->b_in; p.w_out = c->w_out; p.b_out = c->b_out; p.v = c->v; p.h = c->h;
  p.o = static_cast<__nv_bfloat16*>(c->o);
  p.act = static_cast<__nv_bfloat16*>(c->act);
  int rc;
  const size_t R = kStepMaxRows;
  if ((rc = dalloc_t(c, &p.acc_qkv, R * c->qkvd)) || (rc = dalloc_t(c, &p.acc_o, R * W)) ||
      (rc = dalloc_t(c, &p.acc_gu, R * 2 * F)) || (rc = dalloc_t(c, &p.acc_d, R * W)))
    return rc;
  std::vector<const void*> wl;
  for (const LayerW& w : c->L) wl.insert(wl.end(), {w.wqkv.w, w.wo.w, w.wgu.w, w.wd.w});
  void* wd = nullptr;
  if ((rc = dalloc(c, &wd, wl.size() * sizeof(void*)))) return rc;
  if (cudaMemcpy(wd, wl.data(), wl.size() * sizeof(void*), cudaMemcpyHostToDevice) != cudaSuccess)
    return fail(c, UAD_ECUDA, "weight table copy failed");
  p.wl = static_cast<const void* const*>(wd);
  p.q = t.q; p.kcache = t.kcache; p.vtcache = t.vtcache;
  const size_t parts = (size_t)c->step_bmax * a.n_kv_heads * p.n_chunks * t.r_pad;
  if ((rc = dalloc_t(c, &p.part_o, parts * a.head_dim)) || (rc = dalloc_t(c, &p.part_ml, parts * 2))) return rc;
  p.rope_cs = c->rope_cs;
  if ((rc = dalloc_t(c, &p.sync, step_sync_words(L)))) return rc;
  // projection input rows z: tokens, then the step's shift rows (a tensor map of all 64 rows)
  void* z = nullptr;
  if ((rc = dalloc(c, &z, (size_t)kStepMaxRows * W * 2))) return rc;
  p.z = static_cast<__nv_bfloat16*>(z);
  if ((rc = make_tmap(c, z, W, kStepMaxRows))) return rc;
  p.err = c->dev_err;
  c->smaps.z = c->tmaps.at(z);
  c->smaps.o = c->tmaps.at(c->o);
  c->smaps.act = c->tmaps.at(c->act);
  c->smaps.q = c->atmaps.q;
  c->smaps.k = c->atmaps.k2;
  c->smaps.vt = c->atmaps.vt;
  double params = (double)W * a.action_dim * 2;
  params += (double)L * ((double)c->qkvd * W + (double)W * c->qd + 2.0 * F * W + (double)W * F);
  c->step_bytes_w = 2.0 * params;
  c->step_flops_w = 2.0 * params;
  c->step_ok = true;
  return UAD_OK;
}

bool step_path(const uad_ctx* c, int B) { return c->step_ok && !c->step_failed && B <= c->step_bmax; }

// Whether a chunk runs on the persistent kernel: it serves the batch and every step has room
// for its distinct flow times next to the tokens (set by the host plan).
bool chunk_uses_step(const uad_ctx* c, int B, int max_shift) {
  return step_path(c, B) && max_shift <= kStepMaxShift && B * c->a.chunk_len + max_shift <= kStepMaxRows;
}

// Enqueue every kernel of one chunk (begin + n_steps evaluations) for B robots.
void enqueue_chunk(uad_ctx* c, int B, int n_steps, bool step, cudaStream_t s) {
  const uad_arch& a = c->a;
  const int H = a.chunk_len, D = a.action_dim, W = a.width, M = B * H, F = a.mlp_dim;
  const int dt = a.dtype;
  const PlanLayout PL = plan_layout(n_steps, B, H, D);
  const PlanTok* plan = reinterpret_cast<const PlanTok*>(c->plan_dev + PL.plan);
  const int* tau = reinterpret_cast<const int*>(c->plan_dev + PL.tau);
  const int W6 = 6 * W;
  const bool dit = a.kind == UAD_KIND_DIT;

  { Mark mk(c, s, "begin", 12.0 * M * D, 0); launch_begin(c->noise, c->x, c->g, c->u, M * D, c->nonfinite, c->evals, c->stamps, s); }
  if (step) {
    // the persistent kernel's accumulators are zero between uses; clearing them per chunk keeps
    // a chunk that ended in an error from leaking into the next one
    const StepArgs& p = c->st0;
    const size_t R = kStepMaxRows;
    cudaMemsetAsync(p.acc_qkv, 0, R * c->qkvd * 4, s);
    cudaMemsetAsync(p.acc_o, 0, R * W * 4, s);
    cudaMemsetAsync(p.acc_gu, 0, R * 2 * F * 4, s);
    cudaMemsetAsync(p.acc_d, 0, R * W * 4, s);
  }
  PendingResid pend;
  for (int k = 1; k <= n_steps; ++k) {
    const int* tr = tau + (size_t)(k - 1) * M;
    // step epilogue (Euler, TR, release, GAC): its own kernel, or the persistent kernel's end
    EulerArgs ea;
    ea.B = B; ea.H = H; ea.D = D; ea.k = k;
    ea.plan = plan + (size_t)(k - 1) * M;
    ea.gstep = reinterpret_cast<const float*>(c->plan_dev + PL.gstep);
    ea.last_step = reinterpret_cast<const int*>(c->plan_dev + PL.last);
    ea.tail_count = reinterpret_cast<const int*>(c->plan_dev + PL.tailc);
    ea.tail_flag = reinterpret_cast<const int*>(c->plan_dev + PL.tailf);
    ea.gac_mask = c->plan_dev + PL.mask;
    ea.epoch = reinterpret_cast<const int*>(c->plan_dev + PL.epoch);
    ea.rot_dim = reinterpret_cast<const int*>(c->plan_dev + PL.rot);
    ea.v = c->v; ea.x = c->x; ea.g = c->g; ea.u = c->u; ea.rel = c->rel;
    ea.final_out = c->fin; ea.ghost_out = c->ghost; ea.E_out = c->E;
    ea.host_rel = c->host_rel_dev; ea.host_flags = c->host_flags_dev;
    ea.nonfinite = c->nonfinite; ea.evals = c->evals; ea.stamps = c->stamps;
    if (step) {
      StepArgs p = c->st0;
      p.M = M; p.B = B; p.tau_row = tr;
      p.eu = ea;
      p.wait_ns = c->wait_ns;
      p.unreachable = (unsigned)c->test_unreachable;
      p.sidx = reinterpret_cast<const int*>(c->plan_dev + PL.sidx) + (size_t)(k - 1) * M;
      p.sinfo = reinterpret_cast<const int*>(c->plan_dev + PL.sinfo) + (size_t)(k - 1) * (1 + kStepMaxShift);
      cudaMemsetAsync(p.sync, 0, step_sync_words(a.n_layers) * 4, s);
      const double kv = 2.0 * B * a.n_layers * a.n_kv_heads * (double)p.n_keys * a.head_dim * 2;
      const double by = c->step_bytes_w + kv + 16.0 * a.n_layers * M * W + 8.0 * M * D;
      const double fl = c->step_flops_w * M + 4.0 * M * a.n_heads * (double)p.n_keys * a.head_dim * a.n_layers;
      Mark mk(c, s, "step_kernel", by, fl);
      if (launch_step(c->smaps, p, c->sms, s)) fail(c, UAD_ECUDA, "step kernel launch failed");
    } else {
      GemmArgs gi;
      gi.A = c->u; gi.lda = D; gi.a_dtype = F32; gi.w_dtype = dt;
      gi.M = M; gi.N = W; gi.K = D; gi.epi = EPI_STORE; gi.out = c->h; gi.ldo = W; gi.bias = c->b_in;
      if (dit) { gi.add_rows = c->pos_code; gi.add_mod = H; }
      { Mark mk(c, s, "in_proj", gemm_bytes(gi, c->es), 2.0 * M * W * D); gemm(c, c->w_in, gi, s); }
      if (a.kind == UAD_KIND_CONCAT) {
        // the input MLP over [action embedding ; time embedding] (App. C.1, SmolVLA): the time
        // half e(tau) W_it + b_it is a table slice per flow time
        launch_convert(c->h, F32, c->y, dt, (long long)M * W, s);
        GemmArgs ga;
        ga.A = c->y; ga.lda = W; ga.a_dtype = dt; ga.w_dtype = dt;
        ga.M = M; ga.N = W; ga.K = W; ga.epi = EPI_STORE; ga.out = c->h; ga.ldo = W; ga.out_dtype = F32;
        { Mark mk(c, s, "in_mlp_a", gemm_bytes(ga, c->es), 2.0 * M * W * W); gemm(c, c->w_ia, ga, s); }
        { Mark mk(c, s, "in_mlp_silu", 12.0 * M * W, 0); launch_add_tau_silu(c->h, c->tab, c->rowlen, concat_off(c), tr, M, W, c->y, dt, s); }
        GemmArgs go;
        go.A = c->y; go.lda = W; go.a_dtype = dt; go.w_dtype = dt;
        go.M = M; go.N = W; go.K = W; go.epi = EPI_STORE; go.out = c->h; go.ldo = W; go.out_dtype = F32; go.bias = c->b_io;
        { Mark mk(c, s, "in_mlp_out", gemm_bytes(go, c->es), 2.0 * M * W * W); gemm(c, c->w_io, go, s); }
      }
      for (int l = 0; l < a.n_layers; ++l) {
        const LayerW& w = c->L[l];
        const int base = l * W6;
        NormArgs na;
        na.h = c->h; na.ldh = W; na.M = M; na.W = W; na.layer_norm = dit; na.tab = c->tab;
        na.stride = c->rowlen; na.tau_row = tr; na.out = c->y; na.ldo = W; na.out_dtype = dt;
        na.scale_off = dit ? base + W : base;
        na.shift_off = dit ? base : base + W;
        norm_after(c, na, &pend, s);
        GemmArgs gq;
        gq.A = c->y; gq.lda = W; gq.a_dtype = dt; gq.w_dtype = dt;
        gq.M = M; gq.N = c->qkvd; gq.K = W; gq.out = c->qkv; gq.ldo = c->qkvd; gq.out_dtype = dt;
        if (c->attn_tc) {
          QkvTcOut& o = gq.qkv;
          gq.epi = EPI_QKV_TC;
          o.q = c->at0.q; o.kcache = c->at0.kcache; o.vtcache = c->at0.vtcache;
          o.rope = a.rope ? c->rope_cs : nullptr;
          o.H = H; o.P = a.prefix_len; o.NK = c->at0.n_keys; o.NKp = c->at0.nk_pad; o.dh = a.head_dim;
          o.G = a.n_heads / a.n_kv_heads; o.Hkv = a.n_kv_heads; o.L = a.n_layers; o.layer = l;
          o.qd = c->qd; o.kvd = c->kvd;
        }
        { Mark mk(c, s, "qkv_proj", gemm_bytes(gq, c->es), 2.0 * M * gq.N * W); gemm(c, w.wqkv, gq, s); }
        AttnArgs at;
        at.n_heads = a.n_heads; at.n_kv_heads = a.n_kv_heads; at.head_dim = a.head_dim; at.H = H; at.B = B;
        at.q = c->qkv; at.q_ld = c->qkvd;
        at.kc = static_cast<const char*>(c->qkv) + (size_t)c->qd * c->es;
        at.vc = static_cast<const char*>(c->qkv) + (size_t)(c->qd + c->kvd) * c->es;
        at.kc_ld = c->qkvd;
        at.out = c->o; at.out_ld = c->qd; at.dtype = dt; at.scale = 1.f / std::sqrt((float)a.head_dim);
        at.split_ws = c->few_ws; at.split_ctr = c->few_ctr;
        if (!dit) {
          at.kp = static_cast<const char*>(c->kpre) + (size_t)l * a.prefix_len * c->kvd * c->es;
          at.vp = static_cast<const char*>(c->vpre) + (size_t)l * a.prefix_len * c->kvd * c->es;
          at.P = a.prefix_len; at.kp_bstride = (long long)a.n_layers * a.prefix_len * c->kvd;
          at.kp_ld = c->kvd; at.rope_cs = a.rope ? c->rope_cs : nullptr;
        }
        if (c->attn_tc) {
          AttnTcArgs t = c->at0;
          t.batch = B; t.layer = l;
          const double keys = (double)t.n_keys;
          const double by = 2.0 * ((double)B * t.n_keys * c->kvd * 2 + (double)M * 2 * c->qd);
          Mark mk(c, s, "attention", by, 4.0 * M * a.n_heads * keys * a.head_dim);
          launch_attn_tc(c->atmaps, t, s);
        } else {
          const double keys = (double)(at.P + H);
          const double by = c->es * ((double)B * at.P * c->kvd * 2 + (double)M * (2 * c->qd + 2 * c->kvd));
          Mark mk(c, s, dit ? "self_attn" : "attention", by, 4.0 * M * a.n_heads * keys * a.head_dim);
          launch_attention(at, s);
        }
        GemmArgs go;
        go.A = c->o; go.lda = c->qd; go.a_dtype = dt; go.w_dtype = dt;
        go.M = M; go.N = W; go.K = c->qd; go.tau_row = tr;
        resid_gemm(c, w.wo, go, base + 2 * W, nullptr, &pend, "o_proj", s);
        if (dit) {
          NormArgs nc = na;
          nc.tab = nullptr;
          norm_after(c, nc, &pend, s);
          GemmArgs gc;
          gc.A = c->y; gc.lda = W; gc.a_dtype = dt; gc.w_dtype = dt;
          gc.M = M; gc.N = c->qd; gc.K = W; gc.out = c->qc; gc.ldo = c->qd; gc.out_dtype = dt;
          { Mark mk(c, s, "q_cross_proj", gemm_bytes(gc, c->es), 2.0 * M * c->qd * W); gemm(c, w.wqc, gc, s); }
          AttnArgs ac;
          ac.n_heads = a.n_heads; ac.n_kv_heads = a.n_heads; ac.head_dim = a.head_dim; ac.H = H; ac.B = B;
          ac.q = c->qc; ac.q_ld = c->qd;
          ac.kp = static_cast<const char*>(c->kpre) + (size_t)l * a.prefix_len * c->qd * c->es;
          ac.vp = static_cast<const char*>(c->vpre) + (size_t)l * a.prefix_len * c->qd * c->es;
          ac.P = a.prefix_len; ac.kp_bstride = (long long)a.n_layers * a.prefix_len * c->qd; ac.kp_ld = c->qd;
          ac.out = c->o; ac.out_ld = c->qd; ac.dtype = dt; ac.scale = at.scale;
          ac.split_ws = c->few_ws; ac.split_ctr = c->few_ctr;
          {
            const double by = c->es * ((double)B * ac.P * c->qd * 2 + 2.0 * M * c->qd);
            Mark mk(c, s, "cross_attn", by, 4.0 * M * a.n_heads * (double)ac.P * a.head_dim);
            launch_attention(ac, s);
          }
          GemmArgs gco;
          gco.A = c->o; gco.lda = c->qd; gco.a_dtype = dt; gco.w_dtype = dt;
          gco.M = M; gco.N = W; gco.K = c->qd; gco.tau_row = tr;
          resid_gemm(c, w.woc, gco, -1, nullptr, &pend, "o_cross_proj", s);
        }
        NormArgs n2 = na;
        n2.scale_off = dit ? base + 4 * W : base + 3 * W;
        n2.shift_off = dit ? base + 3 * W : base + 4 * W;
        norm_after(c, n2, &pend, s);
        GemmArgs g1;
        g1.A = c->y; g1.lda = W; g1.a_dtype = dt; g1.w_dtype = dt; g1.M = M; g1.K = W;
        g1.out = c->act; g1.ldo = F; g1.out_dtype = dt;
        if (dit) { g1.N = F; g1.epi = EPI_BIAS_GELU; g1.bias = w.b1; }
        else { g1.N = 2 * F; g1.epi = EPI_GEGLU; }
        { Mark mk(c, s, dit ? "mlp_up" : "gate_up_proj", gemm_bytes(g1, c->es), 2.0 * M * g1.N * W); gemm(c, dit ? w.w1 : w.wgu, g1, s); }
        GemmArgs g2;
        g2.A = c->act; g2.lda = F; g2.a_dtype = dt; g2.w_dtype = dt;
        g2.M = M; g2.N = W; g2.K = F; g2.tau_row = tr;
        resid_gemm(c, dit ? w.w2 : w.wd, g2, base + 5 * W, dit ? w.b2 : nullptr, &pend, dit ? "mlp_down" : "down_proj", s);
      }
      NormArgs nf;
      nf.h = c->h; nf.ldh = W; nf.M = M; nf.W = W; nf.layer_norm = dit; nf.tab = c->tab;
      nf.stride = c->rowlen; nf.tau_row = tr; nf.out = c->y; nf.ldo = W; nf.out_dtype = dt;
      nf.scale_off = a.n_layers * W6 + (dit ? W : 0);
      nf.shift_off = a.n_layers * W6 + (dit ? 0 : W);
      norm_after(c, nf, &pend, s);
      GemmArgs go;
      go.A = c->y; go.lda = W; go.a_dtype = dt; go.w_dtype = dt;
      go.M = M; go.N = D; go.K = W; go.out = c->v; go.ldo = D; go.bias = c->b_out;
      {
        Mark mk(c, s, "out_proj", gemm_bytes(go, c->es), 2.0 * M * W * D);
        if (c->w_out_tc.tiled) {
          // on the tensor cores: the weight padded to 128 rows, only the first D stored
          go.N = 128;
          go.n_store = D;
          gemm(c, c->w_out_tc, go, s);
        } else {
          gemm(c, c->w_out, go, s);
        }
      }
    }
    if (!step) { Mark mk(c, s, "euler_tr_gac", 40.0 * M * D, 0); launch_euler(ea, s); }
  }
}

int launches_per_step(const uad_ctx* c, int B) {
  const uad_arch& a = c->a;
  if (step_path(c, B)) return 1;   // persistent evaluation kernel with the step epilogue at its end
  if (a.kind == UAD_KIND_DIT) return 11 * a.n_layers + 4;
  // per layer: norm, qkv, attention (split-KV + combine, or the one-pass kernel), o, norm,
  // gate/up, down
  int attn = 1;
  if (c->attn_tc) {
    AttnTcArgs t = c->at0;
    t.batch = B;
    attn = attn_tc_use_two_pass(t) ? 1 : 2;
  }
  return (6 + attn) * a.n_layers + 4 + (a.kind == UAD_KIND_CONCAT ? 4 : 0);
}

}  // namespace

// =========================================================================================
extern "C" {

const char* uad_version(void) { return "uad-gb300 0.1 (sm_103a)"; }

const char* uad_last_error(const uad_ctx* c) { return c ? c->err.c_str() : "null context"; }

int uad_plan_step(const int32_t* budgets, int32_t H, int32_t k, int32_t tr, int32_t* flags,
                  int32_t* tau_num, int32_t* tau_den) {
  if (!budgets || H < 1 || k < 1 || !flags || !tau_num || !tau_den) return UAD_EINVAL;
  int ns = 0;
  for (int i = 0; i < H; ++i) {
    if (budgets[i] < 1 || budgets[i] > UAD_MAX_STEPS) return UAD_EINVAL;
    ns = std::max(ns, (int)budgets[i]);
  }
  for (int i = 0; i < H; ++i) {
    int f;
    std::pair<int, int> t;
    plan_token(k, budgets[i], ns, tr != 0, &f, &t);
    // public encoding: bit0 active, bit1 ghost, bit2 release, bit3 early, bit4 frozen
    flags[i] = f & (PF_ACTIVE | PF_GHOST | PF_RELEASE | PF_EARLY | PF_FROZEN);
    tau_num[i] = t.first;
    tau_den[i] = t.second;
  }
  return ns;
}

int uad_init(const uad_arch* arch, const float* weights, size_t n_floats, uad_ctx** out) {
  if (!arch || !weights || !out) return UAD_EINVAL;
  *out = nullptr;
  std::string why;
  if (validate_arch(*arch, why) != UAD_OK) {
    fprintf(stderr, "uad_init: invalid arch: %s\n", why.c_str());
    return UAD_EINVAL;
  }
  const std::vector<Tensor> lay = blob_layout(*arch);
  const size_t total = lay.back().off + (size_t)(lay.back().rows * lay.back().cols);
  if (n_floats != total) {
    fprintf(stderr, "uad_init: weight blob has %zu floats, arch needs %zu\n", n_floats, total);
    return UAD_EINVAL;
  }
  uad_ctx* c = new uad_ctx();
  c->a = *arch;
  const uad_arch& a = c->a;
  {
    const char* e = getenv("UAD_GRAPHS");
    if (e && e[0] == '0') c->use_graphs = false;
    e = getenv("UAD_GEMM");
    if (e && !strcmp(e, "simt")) c->force_simt = true;
    e = getenv("UAD_STEP");
    if (e && e[0] == '0') c->step_off = true;
  }
  int rc = UAD_OK;
#define TRY(x)                        \
  do {                                \
    if ((rc = (x)) != UAD_OK) {       \
      fprintf(stderr, "uad_init: %s\n", c->err.c_str()); \
      uad_destroy(c);                 \
      return rc;                      \
    }                                 \
  } while (0)
  if (cudaGetDevice(&c->dev) != cudaSuccess) {
    delete c;
    return UAD_ECUDA;
  }
  cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, c->dev);
  const int W = a.width, D = a.action_dim, F = a.mlp_dim, H = a.chunk_len, dt = a.dtype;
  c->es = dt == BF16 ? 2 : 4;
  c->qd = a.n_heads * a.head_dim;
  c->kvd = a.n_kv_heads * a.head_dim;
  c->qkvd = a.kind == UAD_KIND_DIT ? 3 * c->qd : c->qd + 2 * c->kvd;
  c->rowlen = a.n_layers * 6 * W + 2 * W + (a.kind == UAD_KIND_CONCAT ? W : 0);
  c->mmax = a.max_batch * H;
  const int es = c->es;

  // ---- weights: stage the fp32 blob on the device, then re-lay out each tensor ----
  float* blob = nullptr;
  TRY(dalloc_t(c, &blob, total));
  if (cudaMemcpy(blob, weights, total * 4, cudaMemcpyDefault) != cudaSuccess) {
    fail(c, UAD_ECUDA, "weight upload failed");
    TRY(UAD_ECUDA);
  }
  std::map<std::string, const Tensor*> T;
  for (const Tensor& t : lay) T[t.name] = &t;
  auto src = [&](const std::string& n) { return blob + T.at(n)->off; };
  cudaStream_t s0 = nullptr;
  // linear [K][N] -> library [N][K] (dst rows n*mult + off)
  auto lin = [&](const std::string& n, void* dst, int mult, long long off) {
    launch_relayout(src(n), (int)T.at(n)->rows, (int)T.at(n)->cols, dst, dt, mult, off, s0);
  };
  auto vec = [&](const std::string& n, float** dst) -> int {
    int r = dalloc_t(c, dst, (size_t)T.at(n)->cols);
    if (r) return r;
    return cudaMemcpy(*dst, src(n), T.at(n)->cols * 4, cudaMemcpyDeviceToDevice) == cudaSuccess
               ? UAD_OK : fail(c, UAD_ECUDA, "copy %s", n.c_str());
  };
  const bool concat = a.kind == UAD_KIND_CONCAT;
  if (concat) {
    // no time MLP and no modulation: zero weights, and biases scale = shift = 0, gate = 1, so
    // that the adaptive norms are plain RMSNorm and the residuals ungated
    void* p;
    TRY(dalloc(c, &p, (size_t)W * W * es)); c->t_w1 = (float*)p;
    TRY(dalloc(c, &p, (size_t)W * W * es)); c->t_w2 = (float*)p;
    TRY(dalloc_t(c, &c->t_b1, (size_t)W)); TRY(dalloc_t(c, &c->t_b2, (size_t)W));
    TRY(dalloc(c, &c->w_in, (size_t)W * D * es)); lin("in_w", c->w_in, 1, 0);
    TRY(vec("in_b", &c->b_in));
    TRY(dalloc(c, &c->w_out, (size_t)W * D * es)); lin("out_w", c->w_out, 1, 0);
    TRY(vec("out_b", &c->b_out));
    TRY(dalloc(c, &c->w_mod, (size_t)c->rowlen * W * es));
    TRY(dalloc_t(c, &c->b_mod, (size_t)c->rowlen));
    std::vector<float> bm((size_t)c->rowlen, 0.f);
    for (int l = 0; l < a.n_layers; ++l)
      for (int half = 0; half < 2; ++half)
        std::fill(bm.begin() + (size_t)l * 6 * W + half * 3 * W + 2 * W, bm.begin() + (size_t)l * 6 * W + half * 3 * W + 3 * W, 1.f);
    CK(cudaMemcpy(c->b_mod, bm.data(), bm.size() * 4, cudaMemcpyHostToDevice));
    TRY(dalloc(c, &c->w_it, (size_t)W * W * es)); lin("ti_wt", c->w_it, 1, 0);
    TRY(vec("ti_b", &c->b_it));
    TRY(vec("to_b", &c->b_io));
  } else {
    void* p;
    TRY(dalloc(c, &p, (size_t)W * W * es)); c->t_w1 = (float*)p; lin("t_w1", p, 1, 0);
    TRY(dalloc(c, &p, (size_t)W * W * es)); c->t_w2 = (float*)p; lin("t_w2", p, 1, 0);
    TRY(vec("t_b1", &c->t_b1)); TRY(vec("t_b2", &c->t_b2));
    TRY(dalloc(c, &c->w_in, (size_t)W * D * es)); lin("in_w", c->w_in, 1, 0);
    TRY(vec("in_b", &c->b_in));
    TRY(dalloc(c, &c->w_out, (size_t)W * D * es)); lin("out_w", c->w_out, 1, 0);
    TRY(vec("out_b", &c->b_out));
    // all modulation Linears stacked: rows [layer l: 6W][final: 2W]
    TRY(dalloc(c, &c->w_mod, (size_t)c->rowlen * W * es));
    TRY(dalloc_t(c, &c->b_mod, (size_t)c->rowlen));
    for (int l = 0; l < a.n_layers; ++l) {
      const std::string p = "l" + std::to_string(l) + ".";
      const long long base = (long long)l * 6 * W;
      if (a.kind == UAD_KIND_ADARMS) {
        lin(p + "mod1_w", c->w_mod, 1, base);
        lin(p + "mod2_w", c->w_mod, 1, base + 3 * W);
        CK(cudaMemcpy(c->b_mod + base, src(p + "mod1_b"), 3 * W * 4, cudaMemcpyDeviceToDevice));
        CK(cudaMemcpy(c->b_mod + base + 3 * W, src(p + "mod2_b"), 3 * W * 4, cudaMemcpyDeviceToDevice));
      } else {
        lin(p + "mod_w", c->w_mod, 1, base);
        CK(cudaMemcpy(c->b_mod + base, src(p + "mod_b"), 6 * W * 4, cudaMemcpyDeviceToDevice));
      }
    }
    lin("modf_w", c->w_mod, 1, (long long)a.n_layers * 6 * W);
    CK(cudaMemcpy(c->b_mod + (size_t)a.n_layers * 6 * W, src("modf_b"), 2 * W * 4, cudaMemcpyDeviceToDevice));
  }
  c->L.resize(a.n_layers);
  // allocate a projection in the layout its GEMM uses
  auto mklin = [&](Lin* l, int N, int K) -> int {
    l->N = N; l->K = K;
    l->tiled = dt == BF16 && !c->force_simt && N % 128 == 0 && K % 64 == 0;
    return dalloc(c, &l->w, (size_t)N * K * es);
  };
  auto put = [&](const std::string& n, const Lin& l, int mult, long long off, int rope_dh = 0) {
    if (l.tiled) launch_relayout_tiled(src(n), (int)T.at(n)->rows, (int)T.at(n)->cols, l.w, mult, off, rope_dh, s0);
    else lin(n, l.w, mult, off);
  };
  // tensor-core attention: bf16 joint-attention experts whose QKV projection is tiled (q, k and v
  // each whole 128-row tiles: the projection's epilogue writes each tile in one layout)
  c->attn_tc = a.kind != UAD_KIND_DIT && dt == BF16 && !c->force_simt && c->qd % 128 == 0 && c->kvd % 128 == 0 &&
              W % 64 == 0 && a.prefix_len + H <= attn_tc_max_keys();
  const int qk_perm = c->attn_tc && a.rope ? a.head_dim : 0;
  // the action-out projection on the tensor cores (D <= 128 rows padded to 128, zero)
  if (D <= 128) {
    TRY(mklin(&c->w_out_tc, 128, W));
    if (c->w_out_tc.tiled) put("out_w", c->w_out_tc, 1, 0);
  }
  for (int l = 0; l < a.n_layers; ++l) {
    const std::string p = "l" + std::to_string(l) + ".";
    LayerW& w = c->L[l];
    TRY(mklin(&w.wqkv, c->qkvd, W));
    put(p + "wq", w.wqkv, 1, 0, qk_perm);
    put(p + "wk", w.wqkv, 1, c->qd, qk_perm);
    put(p + "wv", w.wqkv, 1, c->qd + (a.kind == UAD_KIND_DIT ? c->qd : c->kvd));
    TRY(mklin(&w.wo, W, c->qd)); put(p + "wo", w.wo, 1, 0);
    if (a.kind != UAD_KIND_DIT) {
      TRY(mklin(&w.wgu, 2 * F, W));
      put(p + "wg", w.wgu, 2, 0);
      put(p + "wu", w.wgu, 2, 1);
      TRY(mklin(&w.wd, W, F)); put(p + "wd", w.wd, 1, 0);
    } else {
      TRY(mklin(&w.wqc, c->qd, W)); put(p + "wqc", w.wqc, 1, 0);
      TRY(mklin(&w.woc, W, c->qd)); put(p + "woc", w.woc, 1, 0);
      TRY(dalloc(c, &w.wkc, (size_t)c->qd * a.prefix_width * es)); lin(p + "wkc", w.wkc, 1, 0);
      TRY(dalloc(c, &w.wvc, (size_t)c->qd * a.prefix_width * es)); lin(p + "wvc", w.wvc, 1, 0);
      TRY(mklin(&w.w1, F, W)); put(p + "w1", w.w1, 1, 0);
      TRY(mklin(&w.w2, W, F)); put(p + "w2", w.w2, 1, 0);
      TRY(vec(p + "b1", &w.b1)); TRY(vec(p + "b2", &w.b2));
    }
  }
  if (concat) {
    TRY(mklin(&c->w_ia, W, W)); put("ti_wa", c->w_ia, 1, 0);
    TRY(mklin(&c->w_io, W, W)); put("to_w", c->w_io, 1, 0);
  }
  if (cudaDeviceSynchronize() != cudaSuccess || cudaGetLastError() != cudaSuccess) {
    fail(c, UAD_ECUDA, "weight re-layout failed");
    TRY(UAD_ECUDA);
  }
  cudaFree(blob);
  c->allocs.erase(std::find(c->allocs.begin(), c->allocs.end(), (void*)blob));

  // ---- tables ----
  c->tab_cap = 256;
  TRY(dalloc_t(c, &c->tab, (size_t)c->tab_cap * c->rowlen));
  TRY(dalloc_t(c, &c->temb, (size_t)c->tab_cap * W));
  TRY(dalloc_t(c, &c->tc1, (size_t)c->tab_cap * W));
  TRY(dalloc_t(c, &c->tc2, (size_t)c->tab_cap * W));
  if (a.kind != UAD_KIND_DIT && a.rope) {
    const int dh = a.head_dim, half = dh / 2;
    std::vector<float> cs((size_t)H * dh);
    for (int i = 0; i < H; ++i)
      for (int j = 0; j < half; ++j) {
        const double ang = (double)(a.prefix_len + i) * std::pow(10000.0, -2.0 * j / dh);
        cs[(size_t)i * dh + 2 * j] = (float)std::cos(ang);
        cs[(size_t)i * dh + 2 * j + 1] = (float)std::sin(ang);
      }
    TRY(dalloc_t(c, &c->rope_cs, cs.size()));
    CK(cudaMemcpy(c->rope_cs, cs.data(), cs.size() * 4, cudaMemcpyHostToDevice));
  }
  if (a.kind == UAD_KIND_DIT) {
    std::vector<float> pe((size_t)H * W);
    for (int i = 0; i < H; ++i) sinusoid_row((double)i, W, 1.0, &pe[(size_t)i * W]);
    TRY(dalloc_t(c, &c->pos_code, pe.size()));
    CK(cudaMemcpy(c->pos_code, pe.data(), pe.size() * 4, cudaMemcpyHostToDevice));
  }

  // ---- prefix, activations, state ----
  const size_t per_robot_kv = (size_t)a.n_layers * a.prefix_len * (a.kind == UAD_KIND_DIT ? c->qd : c->kvd);
  TRY(dalloc(c, &c->kpre, a.max_batch * per_robot_kv * es));
  TRY(dalloc(c, &c->vpre, a.max_batch * per_robot_kv * es));
  c->has_prefix.assign(a.max_batch, 0);
  if (a.dtype == UAD_DTYPE_BF16 && a.head_dim == 64) {
    // few-query attention split over key chunks (self-attention over the chunk, cross-attention
    // over the prefix): partial rows and zeroed arrival counts
    const int keys = std::max(a.chunk_len + (a.kind == UAD_KIND_DIT ? 0 : a.prefix_len), a.prefix_len);
    TRY(dalloc_t(c, &c->few_ws, std::max<size_t>(1, attn_few_ws_floats(a.max_batch, a.n_heads, a.chunk_len, keys))));
    const size_t nctr = std::max<size_t>(1, attn_few_ctr_count(a.max_batch, a.n_heads, a.chunk_len));
    TRY(dalloc_t(c, &c->few_ctr, nctr));
    CK(cudaMemset(c->few_ctr, 0, nctr * sizeof(unsigned)));
  }
  const size_t M = c->mmax;
  TRY(dalloc_t(c, &c->h, M * W));
  TRY(dalloc(c, &c->y, M * W * es));
  TRY(dalloc(c, &c->qkv, M * c->qkvd * es));
  TRY(dalloc(c, &c->qc, M * c->qd * es));
  TRY(dalloc(c, &c->o, M * c->qd * es));
  TRY(dalloc(c, &c->act, M * F * es));
  for (float** p : {&c->v, &c->x, &c->g, &c->u, &c->rel, &c->fin, &c->ghost, &c->noise})
    TRY(dalloc_t(c, p, M * D));
  TRY(dalloc_t(c, &c->dev_err, 1));
  if (c->attn_tc) {
    AttnTcArgs& t = c->at0;
    t.n_layers = a.n_layers; t.n_kv_heads = a.n_kv_heads; t.group = a.n_heads / a.n_kv_heads;
    t.head_dim = a.head_dim; t.H = H; t.prefix = a.prefix_len; t.n_keys = a.prefix_len + H;
    t.nk_pad = (t.n_keys + 7) / 8 * 8; t.rows = t.group * H; t.r_pad = attn_tc_rpad(t.rows);
    t.scale_log2 = 1.4426950408889634f / std::sqrt((float)a.head_dim);
    t.out_ld = c->qd; t.err = c->dev_err;
    const size_t kvz = (size_t)a.max_batch * a.n_layers * a.n_kv_heads;
    const int chunks = attn_tc_chunks(t.n_keys);
    void* p;
    TRY(dalloc(c, &p, (size_t)a.max_batch * a.n_kv_heads * t.rows * a.head_dim * 2)); t.q = (__nv_bfloat16*)p;
    TRY(dalloc(c, &p, kvz * t.n_keys * a.head_dim * 2)); t.kcache = (__nv_bfloat16*)p;
    TRY(dalloc(c, &p, kvz * a.head_dim * t.nk_pad * 2)); t.vtcache = (__nv_bfloat16*)p;
    TRY(dalloc_t(c, &t.part_o, (size_t)a.max_batch * a.n_kv_heads * chunks * t.r_pad * a.head_dim));
    TRY(dalloc_t(c, &t.part_ml, (size_t)a.max_batch * a.n_kv_heads * chunks * t.r_pad * 2));
    t.out = (__nv_bfloat16*)c->o;
    if (attn_tc_prepare(&c->atmaps, t, a.max_batch)) {
      fail(c, UAD_ECUDA, "attention TMA descriptors failed");
      TRY(UAD_ECUDA);
    }
  }
  if (dt == BF16 && !c->force_simt) {
    TRY(make_tmap(c, c->y, W, (int)M));
    TRY(make_tmap(c, c->o, c->qd, (int)M));
    TRY(make_tmap(c, c->act, F, (int)M));
    const size_t maxN = std::max({(size_t)c->qkvd, (size_t)2 * F, (size_t)W});
    TRY(dalloc_t(c, &c->tc_acc, M * maxN));
    TRY(dalloc_t(c, &c->tc_counters, 1 << 16));
    size_t part = 0;
    for (int b = 1; b <= a.max_batch; ++b)
      part = std::max({part, residual_planes(c, b * H, c->qd) * (size_t)b * H * W,
                       residual_planes(c, b * H, F) * (size_t)b * H * W});
    TRY(dalloc_t(c, &c->part, part));
    gemm_tc_prepare();
  }
  TRY(step_setup(c));
  TRY(dalloc_t(c, &c->E, (size_t)a.max_batch * D));
  TRY(dalloc_t(c, &c->nonfinite, 1));
  TRY(dalloc_t(c, &c->evals, 1));
  TRY(dalloc_t(c, &c->stamps, kFlagStride));
  c->plan_bytes_cap = plan_layout(kMaxSteps, a.max_batch, H, D).total;
  TRY(dalloc(c, (void**)&c->plan_dev, c->plan_bytes_cap));
  CK(cudaHostAlloc((void**)&c->plan_host, c->plan_bytes_cap, cudaHostAllocDefault));
  CK(cudaHostAlloc((void**)&c->status_host, sizeof(uad_ctx::ChunkStatus), cudaHostAllocDefault));
  CK(cudaHostAlloc((void**)&c->host_rel, M * D * 4, cudaHostAllocMapped));
  CK(cudaHostGetDevicePointer((void**)&c->host_rel_dev, c->host_rel, 0));
  CK(cudaHostAlloc((void**)&c->host_flags, (size_t)a.max_batch * kFlagStride * 4, cudaHostAllocMapped));
  CK(cudaHostGetDevicePointer((void**)&c->host_flags_dev, c->host_flags, 0));
  memset(c->host_flags, 0, (size_t)a.max_batch * kFlagStride * 4);
  memset(c->host_rel, 0, M * D * 4);
  CK(cudaStreamCreateWithFlags(&c->worker, cudaStreamNonBlocking));
  CK(cudaEventCreateWithFlags(&c->ev_in, cudaEventDisableTiming));
  CK(cudaEventCreateWithFlags(&c->ev_done, cudaEventDisableTiming));
  // attention kernels need more than 48 KB of dynamic shared memory: opt in once, here
  launch_attention_prepare(a.head_dim);
  launch_euler_prepare();
  CK(cudaDeviceSynchronize());
  CK(cudaGetLastError());
#undef TRY
  *out = c;
  return UAD_OK;
}

int uad_set_prefix_kv(uad_ctx* c, int32_t robot, const void* k, const void* v, int32_t prefix_len,
                      int32_t dtype) {
  if (!c) return UAD_EINVAL;
  const uad_arch& a = c->a;
  if (robot < 0 || robot >= a.max_batch) return fail(c, UAD_EINVAL, "robot %d out of range", robot);
  if (prefix_len != a.prefix_len) return fail(c, UAD_EINVAL, "prefix_len %d != arch %d", prefix_len, a.prefix_len);
  if (dtype != UAD_DTYPE_F32 && dtype != UAD_DTYPE_BF16) return fail(c, UAD_EINVAL, "dtype");
  if (!k) return fail(c, UAD_EINVAL, "null prefix");
  if (c->in_flight) return fail(c, UAD_ESTATE, "a chunk is in flight");
  const int ies = dtype == UAD_DTYPE_BF16 ? 2 : 4;
  cudaStream_t s = c->worker;
  if (a.kind != UAD_KIND_DIT && c->attn_tc) {
    if (!v) return fail(c, UAD_EINVAL, "null prefix values");
    const size_t n = (size_t)a.n_layers * a.prefix_len * c->kvd;
    void *tk = nullptr, *tv = nullptr;
    if (cudaMalloc(&tk, n * ies) != cudaSuccess) return fail(c, UAD_ENOMEM, "prefix staging");
    if (cudaMalloc(&tv, n * ies) != cudaSuccess) { cudaFree(tk); return fail(c, UAD_ENOMEM, "prefix staging"); }
    int rc = UAD_OK;
    if (cudaMemcpyAsync(tk, k, n * ies, cudaMemcpyDefault, s) != cudaSuccess ||
        cudaMemcpyAsync(tv, v, n * ies, cudaMemcpyDefault, s) != cudaSuccess)
      rc = UAD_ECUDA;
    else
      launch_kv_prefix(tk, tv, dtype, c->at0, robot, s);
    cudaError_t e = cudaStreamSynchronize(s);
    cudaFree(tk);
    cudaFree(tv);
    if (rc != UAD_OK || e != cudaSuccess || cudaGetLastError() != cudaSuccess)
      return fail(c, UAD_ECUDA, "prefix upload failed");
  } else if (a.kind != UAD_KIND_DIT) {
    if (!v) return fail(c, UAD_EINVAL, "null prefix values");
    const size_t n = (size_t)a.n_layers * a.prefix_len * c->kvd;
    void* tmp = nullptr;
    if (cudaMalloc(&tmp, n * ies) != cudaSuccess) return fail(c, UAD_ENOMEM, "prefix staging");
    int rc = UAD_OK;
    for (int which = 0; which < 2 && rc == UAD_OK; ++which) {
      const void* srcp = which ? v : k;
      void* dst = static_cast<char*>(which ? c->vpre : c->kpre) + (size_t)robot * n * c->es;
      if (cudaMemcpyAsync(tmp, srcp, n * ies, cudaMemcpyDefault, s) != cudaSuccess) rc = UAD_ECUDA;
      else launch_convert(tmp, dtype, dst, a.dtype, (long long)n, s);
    }
    cudaError_t e = cudaStreamSynchronize(s);
    cudaFree(tmp);
    if (rc != UAD_OK || e != cudaSuccess || cudaGetLastError() != cudaSuccess)
      return fail(c, UAD_ECUDA, "prefix upload failed");
  } else {
    if (v) return fail(c, UAD_EINVAL, "DiT takes prefix tokens in k and NULL v");
    const size_t n = (size_t)a.prefix_len * a.prefix_width;
    void *raw = nullptr, *tok = nullptr;
    if (cudaMalloc(&raw, n * ies) != cudaSuccess) return fail(c, UAD_ENOMEM, "prefix staging");
    if (cudaMalloc(&tok, n * c->es) != cudaSuccess) { cudaFree(raw); return fail(c, UAD_ENOMEM, "prefix staging"); }
    cudaMemcpyAsync(raw, k, n * ies, cudaMemcpyDefault, s);
    launch_convert(raw, dtype, tok, a.dtype, (long long)n, s);
    const size_t per_layer = (size_t)a.prefix_len * c->qd;
    for (int l = 0; l < a.n_layers; ++l) {
      for (int which = 0; which < 2; ++which) {
        GemmArgs g;
        g.A = tok; g.lda = a.prefix_width; g.a_dtype = a.dtype;
        g.W = which ? c->L[l].wvc : c->L[l].wkc; g.w_dtype = a.dtype;
        g.M = a.prefix_len; g.N = c->qd; g.K = a.prefix_width; g.out_dtype = a.dtype;
        g.out = static_cast<char*>(which ? c->vpre : c->kpre) +
                ((size_t)robot * a.n_layers * per_layer + (size_t)l * per_layer) * c->es;
        g.ldo = c->qd;
        launch_gemm_simt(g, s);
      }
    }
    cudaError_t e = cudaStreamSynchronize(s);
    cudaFree(raw);
    cudaFree(tok);
    if (e != cudaSuccess || cudaGetLastError() != cudaSuccess) return fail(c, UAD_ECUDA, "prefix projection failed");
  }
  c->has_prefix[robot] = 1;
  return UAD_OK;
}

int uad_prepare_times(uad_ctx* c, int32_t max_budget) {
  if (!c) return UAD_EINVAL;
  if (max_budget < 1 || max_budget > UAD_MAX_STEPS) return fail(c, UAD_EINVAL, "max_budget");
  if (c->in_flight) return fail(c, UAD_ESTATE, "a chunk is in flight");
  std::vector<std::pair<int, int>> need;
  auto want = [&](std::pair<int, int> f) {
    if (!c->tau_row.count(f) && std::find(need.begin(), need.end(), f) == need.end()) need.push_back(f);
  };
  for (int n = 1; n <= max_budget; ++n)
    for (int j = 0; j < n; ++j) want(reduce(j, n));
  want({1, 1});
  int rc = fill_times(c, need, c->worker);
  if (rc) return rc;
  CK(cudaStreamSynchronize(c->worker));
  return UAD_OK;
}

static int denoise_impl(uad_ctx* c, const float* noise, const uad_schedule* sc, int32_t n_star, void* stream,
                        bool profile) {
  if (!c || !noise || !sc || !sc->budgets) return c ? fail(c, UAD_EINVAL, "null argument") : UAD_EINVAL;
  const uad_arch& a = c->a;
  if (c->in_flight) return fail(c, UAD_ESTATE, "previous chunk not finished");
  const int B = sc->batch, H = a.chunk_len, D = a.action_dim;
  if (B < 1 || B > a.max_batch) return fail(c, UAD_EINVAL, "batch %d not in 1..%d", B, a.max_batch);
  const int S = sc->n_exec == 0 ? H : sc->n_exec;
  if (S < 1 || S > H) return fail(c, UAD_EINVAL, "n_exec %d not in 1..H", S);
  if (sc->gac && !sc->tr && !sc->chunk_relative) return fail(c, UAD_EINVAL, "GAC needs TR");
  if (sc->rot_dim != -1 && (sc->rot_dim < 0 || sc->rot_dim > D - 3))
    return fail(c, UAD_EINVAL, "rot_dim %d not -1 or in 0..%d", sc->rot_dim, D - 3);
  for (int b = 0; b < B; ++b)
    if (!c->has_prefix[b]) return fail(c, UAD_EINVAL, "robot %d has no prefix", b);
  std::vector<int> ns(B, 0);
  for (int b = 0; b < B; ++b)
    for (int i = 0; i < H; ++i) {
      const int n = sc->budgets[b * H + i];
      if (n < 1 || n > UAD_MAX_STEPS) return fail(c, UAD_EINVAL, "budget %d out of range", n);
      ns[b] = std::max(ns[b], n);
    }
  const int steps = *std::max_element(ns.begin(), ns.end());
  if (n_star != 0 && n_star != steps) return fail(c, UAD_EINVAL, "n_star %d != max budget %d", n_star, steps);

  // ---- host plan (Sec. 4.2 Eqs. 4-5, Sec. 4.3 Eq. 7) ----
  const int M = B * H;
  const PlanLayout PL = plan_layout(steps, B, H, D);
  unsigned char* hp = c->plan_host;
  PlanTok* plan = reinterpret_cast<PlanTok*>(hp + PL.plan);
  int* taur = reinterpret_cast<int*>(hp + PL.tau);
  std::vector<std::pair<int, int>> taus((size_t)steps * M);
  std::vector<std::pair<int, int>> need;
  for (int k = 1; k <= steps; ++k)
    for (int b = 0; b < B; ++b)
      for (int i = 0; i < H; ++i) {
        const size_t e = (size_t)(k - 1) * M + b * H + i;
        int f;
        plan_token(k, sc->budgets[b * H + i], ns[b], sc->tr != 0, &f, &taus[e]);
        plan[e].flags = f;
        plan[e].dx = 1.0f / (float)sc->budgets[b * H + i];
        if (!c->tau_row.count(taus[e]) && std::find(need.begin(), need.end(), taus[e]) == need.end())
          need.push_back(taus[e]);
      }
  float* gstep = reinterpret_cast<float*>(hp + PL.gstep);
  int* last = reinterpret_cast<int*>(hp + PL.last);
  int* tailc = reinterpret_cast<int*>(hp + PL.tailc);
  int* tailf = reinterpret_cast<int*>(hp + PL.tailf);
  unsigned char* mask = hp + PL.mask;
  for (int b = 0; b < B; ++b) {
    gstep[b] = 1.0f / (float)ns[b];
    last[b] = ns[b];
    bool any_early = false;
    for (int i = 0; i < H; ++i) any_early |= sc->budgets[b * H + i] < ns[b];
    const bool do_gac = sc->gac && !sc->chunk_relative && any_early;
    int cnt = 0;
    for (int i = 0; i < H; ++i) {
      const int t = do_gac && sc->budgets[b * H + i] == ns[b] && i < S;
      tailf[b * H + i] = t;
      cnt += t;
    }
    tailc[b] = cnt;
  }
  for (int d = 0; d < D; ++d) mask[d] = sc->gac_mask ? (sc->gac_mask[d] ? 1 : 0) : 1;
  c->epoch = c->epoch % 1000000000 + 1;
  *reinterpret_cast<int*>(hp + PL.epoch) = c->epoch;
  *reinterpret_cast<int*>(hp + PL.rot) = sc->rot_dim;

  cudaStream_t user = static_cast<cudaStream_t>(stream);
  cudaStream_t s = c->worker;
  CK(cudaEventRecord(c->ev_in, user));
  CK(cudaStreamWaitEvent(s, c->ev_in, 0));
  int rc = fill_times(c, need, s);
  if (rc) return rc;
  for (size_t e = 0; e < taus.size(); ++e) taur[e] = c->tau_row.at(taus[e]);
  // persistent kernel: each step's distinct flow times (their table rows) and each token's index
  int max_shift = 0;
  {
    int* sidx = reinterpret_cast<int*>(hp + PL.sidx);
    int* sinfo = reinterpret_cast<int*>(hp + PL.sinfo);
    for (int k = 0; k < steps; ++k) {
      int* info = sinfo + (size_t)k * (1 + kStepMaxShift);
      int n = 0;
      for (int m = 0; m < M; ++m) {
        const int row = taur[(size_t)k * M + m];
        int j = 0;
        while (j < n && info[1 + j] != row) ++j;
        if (j == n) {
          if (n < kStepMaxShift) info[1 + n] = row;
          ++n;
        }
        sidx[(size_t)k * M + m] = j < kStepMaxShift ? j : 0;
      }
      for (int j = n; j < kStepMaxShift; ++j) info[1 + j] = 0;
      info[0] = std::min(n, kStepMaxShift);
      max_shift = std::max(max_shift, n);
    }
  }
  const bool use_step = chunk_uses_step(c, B, max_shift);
  CK(cudaMemcpyAsync(c->plan_dev, hp, PL.total, cudaMemcpyHostToDevice, s));
  CK(cudaMemcpyAsync(c->noise, noise, (size_t)M * D * 4, cudaMemcpyDefault, s));
  if (c->use_graphs && !profile) {
    const auto key = std::make_tuple(B, steps, use_step ? 1 : 0);
    auto it = c->graphs.find(key);
    if (it == c->graphs.end()) {
      cudaGraph_t g = nullptr;
      CK(cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal));
      enqueue_chunk(c, B, steps, use_step, s);
      cudaError_t e = cudaStreamEndCapture(s, &g);
      if (e != cudaSuccess) return fail(c, UAD_ECUDA, "graph capture failed: %s", cudaGetErrorString(e));
      cudaGraphExec_t ex = nullptr;
      e = cudaGraphInstantiate(&ex, g, 0);
      cudaGraphDestroy(g);
      if (e != cudaSuccess) return fail(c, UAD_ECUDA, "graph instantiate failed: %s", cudaGetErrorString(e));
      it = c->graphs.emplace(key, ex).first;
    }
    CK(cudaGraphLaunch(it->second, s));
  } else if (profile) {
    // capture with an event-record node around every kernel, so that the event times are
    // GPU timestamps between graph nodes (no host launch gaps)
    c->prof_on = true;
    c->prof.clear();
    c->prof_next = 0;
    // create the events before capture
    {
      int need = 2 * (1 + steps * launches_per_step(c, B)) + 8;
      while ((int)c->prof_ev.size() < need) {
        cudaEvent_t e;
        CK(cudaEventCreate(&e));
        c->prof_ev.push_back(e);
      }
    }
    cudaGraph_t g = nullptr;
    CK(cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal));
    enqueue_chunk(c, B, steps, use_step, s);
    cudaError_t e = cudaStreamEndCapture(s, &g);
    c->prof_on = false;
    if (e != cudaSuccess) return fail(c, UAD_ECUDA, "profile capture failed: %s", cudaGetErrorString(e));
    cudaGraphExec_t ex = nullptr;
    e = cudaGraphInstantiate(&ex, g, 0);
    cudaGraphDestroy(g);
    if (e != cudaSuccess) return fail(c, UAD_ECUDA, "profile instantiate failed: %s", cudaGetErrorString(e));
    e = cudaGraphLaunch(ex, s);
    cudaGraphExecDestroy(ex);
    if (e != cudaSuccess) return fail(c, UAD_ECUDA, "profile launch failed: %s", cudaGetErrorString(e));
  } else {
    enqueue_chunk(c, B, steps, use_step, s);
    CK(cudaGetLastError());
  }
  CK(cudaEventRecord(c->ev_done, s));
  CK(cudaStreamWaitEvent(user, c->ev_done, 0));
  c->in_flight = true;
  c->cur_step = use_step;
  c->cur_B = B;
  c->cur_steps = steps;
  c->cur_budgets.assign(sc->budgets, sc->budgets + (size_t)B * H);
  c->cur_nstar = ns;
  return UAD_OK;
}

int uad_denoise(uad_ctx* c, const float* noise, const uad_schedule* sc, int32_t n_star, void* stream) {
  return denoise_impl(c, noise, sc, n_star, stream, false);
}

int uad_profile_chunk(uad_ctx* c, const float* noise, const uad_schedule* sc, uad_kernel_stat* out,
                      int32_t max_stats, int64_t timeout_us) {
  if (!c || !out || max_stats < 1) return c ? fail(c, UAD_EINVAL, "null argument") : UAD_EINVAL;
  int rc = denoise_impl(c, noise, sc, 0, nullptr, true);
  if (rc) return rc;
  rc = uad_finish(c, nullptr, nullptr, nullptr, nullptr, timeout_us);
  if (rc && rc != UAD_ENONFINITE) return rc;
  std::vector<std::string> names;
  std::vector<uad_kernel_stat> st;
  for (const auto& r : c->prof) {
    float ms = 0.f;
    CK(cudaEventElapsedTime(&ms, c->prof_ev[r.ev0], c->prof_ev[r.ev1]));
    size_t j = 0;
    while (j < names.size() && names[j] != r.name) ++j;
    if (j == names.size()) {
      names.push_back(r.name);
      uad_kernel_stat z{};
      snprintf(z.name, sizeof z.name, "%s", r.name);
      st.push_back(z);
    }
    st[j].launches += 1;
    st[j].total_ms += ms;
    st[j].bytes += r.bytes;
    st[j].flops += r.flops;
  }
  const int n = std::min((int)st.size(), (int)max_stats);
  for (int j = 0; j < n; ++j) out[j] = st[j];
  return n;
}

int uad_poll_released(uad_ctx* c, int32_t robot, int32_t min_ready, int64_t timeout_us, float* out,
                      int32_t* ready, int32_t* release_step) {
  if (!c || !out) return UAD_EINVAL;
  if (c->cur_B == 0) return fail(c, UAD_ESTATE, "no chunk started");
  if (robot < 0 || robot >= c->cur_B) return fail(c, UAD_EINVAL, "robot %d not in this chunk", robot);
  const int H = c->a.chunk_len, D = c->a.action_dim;
  if (min_ready > H) return fail(c, UAD_EINVAL, "min_ready %d exceeds the chunk's %d actions", min_ready, H);
  const int ns = c->cur_nstar[robot];
  const int* bud = &c->cur_budgets[(size_t)robot * H];
  const int* flags = c->host_flags + (size_t)robot * kFlagStride;
  const auto t0 = std::chrono::steady_clock::now();
  std::vector<char> done(H, 0);
  int count = 0;
  for (;;) {
    for (int i = 0; i < H; ++i) {
      if (done[i]) continue;
      const int step = bud[i] < ns ? bud[i] : ns;
      if (__atomic_load_n(&flags[step], __ATOMIC_ACQUIRE) == c->epoch) {
        memcpy(out + (size_t)i * D, c->host_rel + ((size_t)robot * H + i) * D, D * 4);
        done[i] = 1;
        ++count;
        if (ready) ready[i] = 1;
        if (release_step) release_step[i] = step;
      }
    }
    if (count >= min_ready || count == H) break;
    const auto el = std::chrono::duration_cast<std::chrono::microseconds>(std::chrono::steady_clock::now() - t0).count();
    if (el >= timeout_us) break;
    std::this_thread::yield();
  }
  if (ready)
    for (int i = 0; i < H; ++i) if (!done[i]) ready[i] = 0;
  if (release_step)
    for (int i = 0; i < H; ++i) if (!done[i]) release_step[i] = 0;
  if (count < min_ready && count < H) return UAD_ETIMEDOUT;
  return count;
}

int uad_finish(uad_ctx* c, float* final_actions, float* ghost, float* gac_error, uad_stats* st,
               int64_t timeout_us) {
  if (!c) return UAD_EINVAL;
  if (!c->in_flight) return fail(c, UAD_ESTATE, "no chunk in flight");
  const auto t0 = std::chrono::steady_clock::now();
  for (;;) {
    cudaError_t e = cudaEventQuery(c->ev_done);
    if (e == cudaSuccess) break;
    if (e != cudaErrorNotReady) return fail(c, UAD_ECUDA, "chunk failed: %s", cudaGetErrorString(e));
    const auto el = std::chrono::duration_cast<std::chrono::microseconds>(std::chrono::steady_clock::now() - t0).count();
    if (timeout_us >= 0 && el >= timeout_us) return fail(c, UAD_ETIMEDOUT, "chunk not finished after %lld us", (long long)el);
    std::this_thread::yield();
  }
  c->in_flight = false;
  // the outputs and the status words as one batch of copies on the (now idle) worker stream and a
  // single wait, so that the GPU idles for one host round trip between chunks, not one per copy
  const size_t n = (size_t)c->cur_B * c->a.chunk_len * c->a.action_dim;
  cudaStream_t s = c->worker;
  uad_ctx::ChunkStatus* cs = c->status_host;
  if (final_actions) CK(cudaMemcpyAsync(final_actions, c->fin, n * 4, cudaMemcpyDefault, s));
  if (ghost) CK(cudaMemcpyAsync(ghost, c->ghost, n * 4, cudaMemcpyDefault, s));
  if (gac_error) CK(cudaMemcpyAsync(gac_error, c->E, (size_t)c->cur_B * c->a.action_dim * 4, cudaMemcpyDefault, s));
  CK(cudaMemcpyAsync(&cs->derr, c->dev_err, 4, cudaMemcpyDeviceToHost, s));
  CK(cudaMemcpyAsync(&cs->nonfinite, c->nonfinite, 4, cudaMemcpyDeviceToHost, s));
  CK(cudaMemcpyAsync(&cs->evals, c->evals, 4, cudaMemcpyDeviceToHost, s));
  CK(cudaMemcpyAsync(cs->stamps, c->stamps, kFlagStride * 8, cudaMemcpyDeviceToHost, s));
  CK(cudaStreamSynchronize(s));
  const int derr = cs->derr, nonfinite = cs->nonfinite, evals = cs->evals;
  if (derr) {
    cudaMemset(c->dev_err, 0, 4);
    if (c->cur_step) {
      // the persistent kernel's grid barriers need all of its CTAs resident at once, which a
      // shared GPU (or one partitioned among processes) may not grant: later chunks run on the
      // per-operation kernels
      c->step_failed = true;
      return fail(c, UAD_ECUDA, "a wait of the persistent kernel timed out (code %d); outputs are not valid; "
                  "later chunks run on the per-operation kernels", derr);
    }
    return fail(c, UAD_ECUDA, "a kernel wait timed out (code %d); outputs are not valid", derr);
  }
  c->last_stamps.assign(cs->stamps, cs->stamps + kFlagStride);
  c->last_steps = c->cur_steps;
  if (st) {
    st->evals = evals;
    st->n_star = c->cur_steps;
    st->nonfinite = nonfinite;
    st->tr_extra_evals = evals - c->cur_steps;
  }
  return nonfinite ? fail(c, UAD_ENONFINITE, "%d non-finite velocity entries", nonfinite) : UAD_OK;
}

int uad_step_times(const uad_ctx* c, double* ms, int32_t max_entries) {
  if (!c || !ms) return UAD_EINVAL;
  const int n = std::min(c->last_steps, (int)max_entries);
  for (int k = 1; k <= n; ++k) ms[k - 1] = (double)(c->last_stamps[k] - c->last_stamps[0]) * 1e-6;
  return n;
}

int uad_launches_per_chunk(const uad_ctx* c, int32_t batch, int32_t n_star) {
  if (!c || batch < 1 || n_star < 1) return UAD_EINVAL;
  return 1 + n_star * launches_per_step(c, batch);
}

int uad_so3_check(const float* w, int32_t n, float* log_exp, float* log_comp) {
  if (!w || !log_exp || !log_comp || n < 1 || n > (1 << 20)) return UAD_EINVAL;
  const size_t bytes = (size_t)n * 3 * 4;
  float* d = nullptr;
  if (cudaMalloc(&d, 3 * bytes) != cudaSuccess) return UAD_ECUDA;
  int rc = UAD_OK;
  if (cudaMemcpy(d, w, bytes, cudaMemcpyHostToDevice) != cudaSuccess) rc = UAD_ECUDA;
  if (!rc) {
    launch_so3_check(d, n, d + 3 * (size_t)n, d + 6 * (size_t)n, nullptr);
    if (cudaGetLastError() != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess ||
        cudaMemcpy(log_exp, d + 3 * (size_t)n, bytes, cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemcpy(log_comp, d + 6 * (size_t)n, bytes, cudaMemcpyDeviceToHost) != cudaSuccess)
      rc = UAD_ECUDA;
  }
  cudaFree(d);
  return rc;
}

int uad_set_wait_limit(uad_ctx* c, int64_t wait_ns, int32_t unreachable) {
  if (!c || wait_ns <= 0 || unreachable < 0) return UAD_EINVAL;
  if (c->in_flight) return fail(c, UAD_ESTATE, "chunk in flight");
  c->wait_ns = (unsigned long long)wait_ns;
  c->test_unreachable = unreachable;
  c->step_failed = false;   // the persistent kernel is tried again
  // the launch arguments are baked into the cached graphs
  for (auto& kv : c->graphs) cudaGraphExecDestroy(kv.second);
  c->graphs.clear();
  return UAD_OK;
}

void uad_destroy(uad_ctx* c) {
  if (!c) return;
  if (c->in_flight && c->ev_done) {
    // bounded wait so that no kernel still writes into memory about to be freed; if the chunk
    // is still running after it, the device memory is deliberately leaked, not freed under it
    const auto t0 = std::chrono::steady_clock::now();
    while (cudaEventQuery(c->ev_done) == cudaErrorNotReady &&
           std::chrono::steady_clock::now() - t0 < std::chrono::seconds(10))
      std::this_thread::yield();
    if (cudaEventQuery(c->ev_done) == cudaErrorNotReady) {
      fprintf(stderr, "uad_destroy: chunk still running; device memory of this context is not freed\n");
      return;
    }
  }
  for (auto& kv : c->graphs) cudaGraphExecDestroy(kv.second);
  for (cudaEvent_t e : c->prof_ev) cudaEventDestroy(e);
  if (c->worker) cudaStreamDestroy(c->worker);
  if (c->ev_in) cudaEventDestroy(c->ev_in);
  if (c->ev_done) cudaEventDestroy(c->ev_done);
  for (void* p : c->allocs) cudaFree(p);
  if (c->plan_host) cudaFreeHost(c->plan_host);
  if (c->status_host) cudaFreeHost(c->status_host);
  if (c->host_rel) cudaFreeHost(c->host_rel);
  if (c->host_flags) cudaFreeHost(c->host_flags);
  delete c;
}

}  // extern "C"
