// Host runtime of the FeatFix cached denoising path and the C ABI of
// include/featfix.h: context and workspace, the fixed schedule (Section 3.3),
// the draft weights of Eq. 2, the per-step block loop (Eqs. 1-5), logs,
// accounting, debug capture, kernel timing and the CUDA-graph replay of
// whole trajectories.
#include "featfix.h"
#include "featfix_ops.h"
#include "ff_common.cuh"

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

using namespace ff;

namespace {

constexpr int NKCLASS = 5;

struct Capture {
  int step, layer;
  void* in;
  void* out;
  void* hist[4];   // history entries the block's draft reads, newest first
  int nhist;
};

struct TimedLaunch {
  cudaEvent_t a, b;
  double work;
};

}  // namespace

struct featfix_ctx {
  featfix_model_desc d;
  DType dt;
  int es;
  int L, Bm, Nt, Ni, Ntot, C, H, hd, M, P, fin, fout;
  long long T, E;
  int gf, gh, gw;
  std::vector<const void*> w;
  cudaStream_t user_st = nullptr;  // caller's stream
  cudaStream_t cap_st = nullptr;   // private stream used only to capture graphs
  cudaStream_t st = nullptr;       // stream work is issued on (user_st, or cap_st while capturing)

  // activations
  void *xa = nullptr, *xb = nullptr, *xm = nullptr, *qkv = nullptr, *att = nullptr, *u1 = nullptr, *big = nullptr;
  void *patches = nullptr, *pos = nullptr;
  float* mout = nullptr;
  float2* rope = nullptr;
  // refresh history: per-block increments R_l and their sum over blocks
  void* ring = nullptr;
  void* sring = nullptr;            // [S][E]: x_L - x_0 of each refresh step
  void* x0buf = nullptr;            // block-0 input of the current step
  void* shadow = nullptr;           // Verify arm: paid check on a copy
  int S = 0;
  // modulation: concatenated block weights and the per-trajectory tables
  void* wmod = nullptr;
  void* bmod = nullptr;
  long long Nblk = 0;
  std::vector<long long> moff;      // column of block l, stream s (0 image / only, 1 text) at 2l + s
  float* d_times = nullptr;         // [steps] model times
  int* d_need = nullptr;            // [steps] row block in the block-mod table, -1 if none
  std::vector<int> need_row;
  int n_need = 0;
  void* sin_tab = nullptr;          // [steps, 256]
  void* thid_tab = nullptr;         // [steps, C]
  float* temb_tab = nullptr;        // [steps, C]
  void* cs_all = nullptr;           // [steps * Bm, C]   SiLU(c)
  void* cs_need = nullptr;          // [n_need * Bm, C]  gathered rows of steps with exact blocks
  float* bmodtab = nullptr;         // [(n_need + 1) * Bm, Nblk]; the last row block is for featfix_debug_block
  float* fmodtab = nullptr;         // [steps * Bm, 2C]
  int mod_row_override = -1;
  // adaLN LayerNorm fused across GEMMs (bf16): the GEMM producing a block
  // input also writes its scaled copy (into xm) and 32-column statistics
  // (lnst); the next layer's GEMM corrects its accumulator per row with the
  // per-sample tables (1 + s) W^T and sh W^T (lncd).  One job per LayerNorm
  // of a block and stream.
  bool lnf = false;
  float2* lnst = nullptr;           // [T, C / 32]
  float* lncd = nullptr;            // per job: [(row blocks) * Bm][2][N]: c row, d row
  void* lnab = nullptr;             // per job: [2 * (row blocks) * Bm][C] operand rows (1 + scale), shift
  int2* d_lnjobs = nullptr;         // per job: columns of its scale and shift chunks in a modulation row
  std::vector<int2> lnjobs;
  std::vector<int> lnjob_n;         // per job: N of the layer after the LayerNorm
  std::vector<const void*> lnjob_w; // per job: that layer's weight
  std::vector<int> lnjob_at;        // (4 l + 2 s + k) -> job, -1 if none (s 0 image / only, 1 text; k 0 qkv, 1 fc1)
  std::vector<long long> lncd_off;  // per job: offset (floats) of its table in lncd
  long long lnab_job = 0;           // elements of one job's operand rows
  int ln_rb = 0;                    // row blocks the tables hold
  bool ln_src[2] = {false, false};  // xm rows of stream s hold the scaled copy for the next LayerNorm
  bool ln_next = false;             // the block being run feeds the next block's first LayerNorm
  // logs
  double* dsums = nullptr;
  int max_logs = 0;
  void* vws = nullptr;
  size_t vws_bytes = 0;
  // device copies of featfix_sample's inputs (fixed addresses for the graph)
  float* g_lat = nullptr;
  void* g_cond = nullptr;
  size_t cond_bytes = 0;
  long long lat_elems = 0;
  float* h_latent = nullptr;        // featfix_sample_host output staging
  void* h_cond = nullptr;

  // schedule
  bool sched = false;
  int steps = 0, K = 0, mode = 0;
  unsigned flags = 0;
  std::vector<unsigned char> kinds;
  std::vector<int> keff;
  std::vector<double> wts;
  std::vector<int> keff_bl;         // per (step, block): FEATFIX_FLAG_SITE_UPDATES_HISTORY
  std::vector<double> wts_bl;
  std::vector<int> bhead;           // per block: ring slot of its newest increment
  int fmask_axis = FEATFIX_MASK_NONE;  // partial forwarding at FeatFix sites
  unsigned char* d_rmask = nullptr;    // [T] per token row (FEATFIX_MASK_TOKENS)
  unsigned char* d_cmask = nullptr;    // [C] per channel (FEATFIX_MASK_CHANNELS)
  std::vector<char> isref;

  // trajectory state
  int next_step = 0;
  int head = 0, count = 0;
  std::vector<std::pair<int, int>> log_sites;
  featfix_counters cnt = {0, 0, 0, 0};
  std::vector<Capture> caps;

  // graph of a whole trajectory
  cudaGraphExec_t gexec = nullptr;
  bool graph_ok = false;
  bool capturing = false;
  long long graph_kernels = 0;
  std::vector<TimedLaunch> gtimed[NKCLASS];

  // kernel timing
  bool timing[NKCLASS] = {false, false, false, false, false};
  std::vector<TimedLaunch> pending[NKCLASS];
  std::vector<cudaEvent_t> evpool;
  double tms[NKCLASS] = {0, 0, 0, 0, 0};
  double twork[NKCLASS] = {0, 0, 0, 0, 0};
  long long tcount[NKCLASS] = {0, 0, 0, 0, 0};

  std::string err;
};

namespace {

featfix_status fail(featfix_ctx* c, featfix_status s, const std::string& msg) {
  if (c) c->err = msg;
  return s;
}

#define FF_CK(call)                                                                                \
  do {                                                                                             \
    cudaError_t e__ = (call);                                                                      \
    if (e__ != cudaSuccess)                                                                        \
      return fail(ctx, FEATFIX_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e__));     \
  } while (0)

#define FF_TRY(call)                          \
  do {                                        \
    featfix_status s__ = (call);              \
    if (s__ != FEATFIX_OK) return s__;        \
  } while (0)

int n_layers(const featfix_model_desc& d) { return d.arch == FEATFIX_ARCH_MMDIT ? d.n_dual + d.n_single : d.n_dual; }

int patch_vol(const featfix_model_desc& d) { return (d.lat_f > 0 ? d.patch_t : 1) * d.patch * d.patch; }

int img_tokens(const featfix_model_desc& d) {
  const int gf = d.lat_f > 0 ? d.lat_f / d.patch_t : 1;
  return gf * (d.lat_h / d.patch) * (d.lat_w / d.patch);
}

std::string check_desc(const featfix_model_desc* d) {
  if (!d) return "null model description";
  if (d->arch != FEATFIX_ARCH_DIT && d->arch != FEATFIX_ARCH_MMDIT) return "unknown arch";
  if (d->n_dual < 0 || d->n_single < 0 || n_layers(*d) < 1) return "no blocks";
  if (d->arch == FEATFIX_ARCH_DIT && (d->n_single != 0 || d->txt_tokens != 0)) return "DiT has no single blocks or text";
  if (d->hidden <= 0 || d->heads <= 0 || d->head_dim <= 0 || d->hidden != d->heads * d->head_dim)
    return "hidden != heads * head_dim";
  if (d->head_dim % 8 || d->head_dim > 128) return "head_dim must be a multiple of 8, <= 128";
  if (d->hidden % 32 || d->mlp <= 0 || d->mlp % 32) return "hidden and mlp must be multiples of 32";
  if (d->hidden > 4096) return "hidden above 4096";
  if (d->in_ch <= 0 || d->out_ch < d->in_ch) return "bad channel counts";
  if (d->patch <= 0 || d->lat_h % d->patch || d->lat_w % d->patch || d->lat_h <= 0 || d->lat_w <= 0)
    return "latent not divisible by patch";
  if (d->lat_f < 0 || (d->lat_f > 0 && (d->patch_t <= 0 || d->lat_f % d->patch_t))) return "bad temporal patch";
  if (d->txt_tokens < 0) return "bad text length";
  if (d->batch <= 0) return "bad batch";
  const int bm = d->batch * (d->cfg ? 2 : 1);
  if (bm > 64) return "model batch above 64";
  if (d->arch == FEATFIX_ARCH_DIT && d->n_classes <= 0) return "DiT needs classes";
  if (d->rope_dims != 0 && d->rope_dims != 2 && d->rope_dims != 3) return "rope_dims must be 0, 2 or 3";
  if (d->rope_dims == 3 && d->lat_f <= 0) return "3-D rotary needs frames";
  if (d->rope_dims != 0 && d->arch != FEATFIX_ARCH_MMDIT) return "rotary positions are for MMDiT";
  if (d->dtype != FEATFIX_DTYPE_F32 && d->dtype != FEATFIX_DTYPE_BF16) return "bad dtype";
  if (d->sampler != FEATFIX_SAMPLER_EULER && d->sampler != FEATFIX_SAMPLER_DDIM) return "bad sampler";
  if (d->arch == FEATFIX_ARCH_DIT && d->hidden % 4) return "position embedding needs hidden % 4 == 0";
  const int fo = patch_vol(*d) * d->out_ch, fi = patch_vol(*d) * d->in_ch;
  const int v = d->dtype == FEATFIX_DTYPE_F32 ? 4 : 8;
  if (fo % v || fi % v) return "patch feature widths must be multiples of the 16-byte vector";
  return "";
}

// ---------------------------------------------------------------------------
// schedule and draft weights
// ---------------------------------------------------------------------------
// Weights w_j of the j-th newest refresh increment so that the draft's
// forecast is sum_j w_j R_{s_j}.
//  default: Lagrange basis of the polynomial through the nodes, evaluated at
//           t -- equal to the Taylor series of Eq. 2 whose derivatives are
//           those of that polynomial at s_0.
//  recursive: Delta^(0)_j = R_j, Delta^(k)_j = (Delta^(k-1)_j -
//           Delta^(k-1)_{j+1}) / (s_j - s_{j+1}), forecast
//           sum_k (t - s_0)^k / k! Delta^(k)_0, expanded over the R_j.
void draft_weights(const std::vector<int>& s, int t, bool recursive, double* w) {
  const int n = (int)s.size();
  for (int j = 0; j < 4; ++j) w[j] = 0.0;
  if (!recursive) {
    for (int j = 0; j < n; ++j) {
      double p = 1.0;
      for (int m = 0; m < n; ++m)
        if (m != j) p *= (double)(t - s[m]) / (double)(s[j] - s[m]);
      w[j] = p;
    }
    return;
  }
  // lvl[j][r]: coefficient of R_r in Delta^(k)_j
  std::vector<std::vector<double>> lvl(n, std::vector<double>(n, 0.0));
  for (int j = 0; j < n; ++j) lvl[j][j] = 1.0;
  double fact = 1.0, pw = 1.0;
  for (int r = 0; r < n; ++r) w[r] += lvl[0][r];
  for (int k = 1; k < n; ++k) {
    std::vector<std::vector<double>> nx(n - k, std::vector<double>(n, 0.0));
    for (int j = 0; j < n - k; ++j)
      for (int r = 0; r < n; ++r) nx[j][r] = (lvl[j][r] - lvl[j + 1][r]) / (double)(s[j] - s[j + 1]);
    lvl.swap(nx);
    fact *= k;
    pw *= (double)(t - s[0]);
    for (int r = 0; r < n; ++r) w[r] += pw / fact * lvl[0][r];
  }
}

// Per step: kinds[i*L + l], the draft order / weights of the refresh-only
// history (keff[i], wts[i*4 + j]) and, per (step, block), those of the
// history a draft of that block actually reads (keff_bl[i*L + l],
// wts_bl[(i*L + l)*4 + j]): the same unless FEATFIX_FLAG_SITE_UPDATES_HISTORY
// lets a site push its block's increment.
featfix_status plan_core(int steps, int L, const int* refresh, int n_refresh, int K, const featfix_site* sites,
                         int n_sites, int mode, unsigned flags, std::vector<unsigned char>& kinds,
                         std::vector<int>& keff, std::vector<double>& wts, std::vector<char>& isref,
                         std::vector<int>& keff_bl, std::vector<double>& wts_bl, std::string& err) {
  if (mode < FEATFIX_MODE_FEATFIX || mode > FEATFIX_MODE_VANILLA) { err = "unknown mode"; return FEATFIX_ERR_INVALID_ARG; }
  if (steps < 1 || L < 1) { err = "steps and layers must be positive"; return FEATFIX_ERR_SCHEDULE; }
  if (K < 0 || K > 3) { err = "draft order must be in [0, 3]"; return FEATFIX_ERR_SCHEDULE; }
  if (n_refresh < 1 || !refresh) { err = "no refresh steps"; return FEATFIX_ERR_SCHEDULE; }
  if (n_sites < 0 || (n_sites > 0 && !sites)) { err = "bad site list"; return FEATFIX_ERR_INVALID_ARG; }
  isref.assign(steps, 0);
  for (int k = 0; k < n_refresh; ++k) {
    const int r = refresh[k];
    if (r < 0 || r >= steps) { err = "refresh step out of range"; return FEATFIX_ERR_SCHEDULE; }
    if (isref[r]) { err = "duplicate refresh step"; return FEATFIX_ERR_SCHEDULE; }
    isref[r] = 1;
  }
  if (!isref[0]) { err = "step 0 must be a full refresh"; return FEATFIX_ERR_SCHEDULE; }
  std::vector<char> issite((size_t)steps * L, 0);
  for (int k = 0; k < n_sites; ++k) {
    const int i = sites[k].step, l = sites[k].layer;
    if (i < 0 || i >= steps || l < 0 || l >= L) { err = "site out of range"; return FEATFIX_ERR_SCHEDULE; }
    if (isref[i]) { err = "site on a refresh step"; return FEATFIX_ERR_SCHEDULE; }
    if (issite[(size_t)i * L + l]) { err = "duplicate site"; return FEATFIX_ERR_SCHEDULE; }
    issite[(size_t)i * L + l] = 1;
  }
  kinds.assign((size_t)steps * L, FEATFIX_PLAN_DRAFT);
  keff.assign(steps, -1);
  wts.assign((size_t)steps * 4, 0.0);
  keff_bl.assign((size_t)steps * L, -1);
  wts_bl.assign((size_t)steps * L * 4, 0.0);
  const bool recursive = (flags & FEATFIX_FLAG_TAYLOR_RECURSIVE) != 0;
  const bool site_push = (flags & FEATFIX_FLAG_SITE_UPDATES_HISTORY) != 0 && mode != FEATFIX_MODE_VANILLA;
  auto push = [K](std::vector<int>& nd, int i) {
    nd.insert(nd.begin(), i);
    if ((int)nd.size() > K + 1) nd.resize(K + 1);
  };
  std::vector<int> nodes;                // refresh steps, newest first
  std::vector<std::vector<int>> bnodes(L);  // per block: refreshes (+ its sites)
  for (int i = 0; i < steps; ++i) {
    if (isref[i]) {
      push(nodes, i);
      for (int l = 0; l < L; ++l) push(bnodes[l], i);
    }
    const bool all_exact = mode == FEATFIX_MODE_VANILLA || isref[i];
    for (int l = 0; l < L; ++l) {
      unsigned char k = FEATFIX_PLAN_DRAFT;
      if (all_exact) k = FEATFIX_PLAN_EXACT;
      else if (issite[(size_t)i * L + l]) k = FEATFIX_PLAN_SITE;
      kinds[(size_t)i * L + l] = k;
    }
    if (!all_exact) {
      const int ke = std::min(K, (int)nodes.size() - 1);
      keff[i] = ke;
      std::vector<int> s(nodes.begin(), nodes.begin() + ke + 1);
      draft_weights(s, i, recursive, &wts[(size_t)i * 4]);
      for (int l = 0; l < L; ++l) {
        const std::vector<int>& nd = bnodes[l];
        const int kb = std::min(K, (int)nd.size() - 1);
        keff_bl[(size_t)i * L + l] = kb;
        std::vector<int> sb(nd.begin(), nd.begin() + kb + 1);
        draft_weights(sb, i, recursive, &wts_bl[((size_t)i * L + l) * 4]);
        // a site's own draft reads the history before its push
        if (site_push && kinds[(size_t)i * L + l] == FEATFIX_PLAN_SITE) push(bnodes[l], i);
      }
    }
  }
  return FEATFIX_OK;
}

// ---------------------------------------------------------------------------
// samplers (host constants)
// ---------------------------------------------------------------------------
double ddim_alpha_bar(int tau) {
  double ab = 1.0;
  for (int k = 0; k <= tau; ++k) ab *= 1.0 - (1e-4 + (0.02 - 1e-4) * (double)k / 999.0);
  return ab;
}

double model_time(const featfix_ctx* c, int i) {
  if (c->d.sampler == FEATFIX_SAMPLER_EULER) return 1000.0 * (1.0 - (double)i / c->steps);
  return (double)(1000 - (1000 / c->steps) * (i + 1));
}

void sampler_coeffs(const featfix_ctx* c, int i, float* c1, float* c2) {
  if (c->d.sampler == FEATFIX_SAMPLER_EULER) {
    *c1 = 1.0f;
    *c2 = (float)((1.0 - (double)(i + 1) / c->steps) - (1.0 - (double)i / c->steps));
    return;
  }
  const int stride = 1000 / c->steps;
  const double at = ddim_alpha_bar(1000 - stride * (i + 1));
  const double ap = i + 1 < c->steps ? ddim_alpha_bar(1000 - stride * (i + 2)) : 1.0;
  *c1 = (float)std::sqrt(ap / at);
  *c2 = (float)(std::sqrt(1.0 - ap) - std::sqrt(ap * (1.0 - at) / at));
}

// ---------------------------------------------------------------------------
// kernel timing: CUDA events on the work stream around each launch of a
// timed kernel class; inside a graph capture the events become external
// event-record nodes that every replay records again.
// ---------------------------------------------------------------------------
cudaEvent_t ev_get(featfix_ctx* c) {
  if (!c->evpool.empty()) {
    cudaEvent_t e = c->evpool.back();
    c->evpool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

struct KTimer {
  featfix_ctx* c;
  int k;
  double work;
  cudaEvent_t a = nullptr;
  KTimer(featfix_ctx* c_, int k_, double work_) : c(c_), k(k_), work(work_) {
    if (!c->timing[k]) return;
    a = ev_get(c);
    if (c->capturing) cudaEventRecordWithFlags(a, c->st, cudaEventRecordExternal);
    else cudaEventRecord(a, c->st);
  }
  ~KTimer() {
    if (!a) return;
    cudaEvent_t b = ev_get(c);
    if (c->capturing) {
      cudaEventRecordWithFlags(b, c->st, cudaEventRecordExternal);
      c->gtimed[k].push_back({a, b, work});
    } else {
      cudaEventRecord(b, c->st);
      c->pending[k].push_back({a, b, work});
    }
  }
};

void timing_drain(featfix_ctx* c) {
  for (int k = 0; k < NKCLASS; ++k) {
    for (auto& t : c->pending[k]) {
      float ms = 0.f;
      if (cudaEventElapsedTime(&ms, t.a, t.b) == cudaSuccess) {
        c->tms[k] += ms;
        c->twork[k] += t.work;
        c->tcount[k] += 1;
      }
      c->evpool.push_back(t.a);
      c->evpool.push_back(t.b);
    }
    c->pending[k].clear();
  }
}

// After a replay (stream synchronised): the graph's events hold that replay's times.
void timing_take_graph(featfix_ctx* c) {
  for (int k = 0; k < NKCLASS; ++k) {
    if (!c->timing[k]) continue;
    for (auto& t : c->gtimed[k]) {
      float ms = 0.f;
      if (cudaEventElapsedTime(&ms, t.a, t.b) == cudaSuccess) {
        c->tms[k] += ms;
        c->twork[k] += t.work;
        c->tcount[k] += 1;
      }
    }
  }
}

void graph_reset(featfix_ctx* c) {
  if (c->gexec) cudaGraphExecDestroy(c->gexec);
  c->gexec = nullptr;
  c->graph_ok = false;
  for (int k = 0; k < NKCLASS; ++k) {
    for (auto& t : c->gtimed[k]) {
      c->evpool.push_back(t.a);
      c->evpool.push_back(t.b);
    }
    c->gtimed[k].clear();
  }
}

// ---------------------------------------------------------------------------
// building blocks
// ---------------------------------------------------------------------------
void* off(void* base, long long elems, int es) { return reinterpret_cast<char*>(base) + elems * es; }
const void* coff(const void* base, long long elems, int es) { return reinterpret_cast<const char*>(base) + elems * es; }

cudaError_t dense(featfix_ctx* c, int M, int N, int K, const void* A, int lda, const void* W, const EpiArgs& e) {
  KTimer tm(c, FEATFIX_KCLASS_GEMM, 2.0 * M * N * (double)K);
  if (c->dt == BF16) return gemm_tc(M, N, K, A, lda, W, K, e, c->st);
  return gemm_simt(c->dt, M, N, K, A, lda, W, K, e, c->st);
}

// Two streams' layers of the same shape (image rows M0, text rows M1) in one
// launch where the tensor-core GEMM can group them.
cudaError_t dense2(featfix_ctx* c, int M0, const void* A0, const void* W0, const EpiArgs& e0, int M1, const void* A1,
                   const void* W1, const EpiArgs& e1, int N, int K, int lda) {
  if (c->dt != BF16) {
    const cudaError_t r = dense(c, M1, N, K, A1, lda, W1, e1);
    return r != cudaSuccess ? r : dense(c, M0, N, K, A0, lda, W0, e0);
  }
  KTimer tm(c, FEATFIX_KCLASS_GEMM, 2.0 * (M0 + M1) * N * (double)K);
  return gemm_tc_grouped(M0, A0, W0, e0, M1, A1, W1, e1, N, K, lda, K, c->st);
}

EpiArgs epi(void* out, int ldo, const void* bias) {
  EpiArgs e = epi_plain(out, ldo);
  e.bias = bias;
  return e;
}

cudaError_t run_attention(featfix_ctx* c, const void* q, const void* k, const void* v, int ld, void* out, int ldo) {
  const double N = c->Ntot;
  KTimer tm(c, FEATFIX_KCLASS_ATTENTION, 4.0 * c->Bm * c->H * N * N * c->hd);
  AttnArgs a;
  a.q = q; a.k = k; a.v = v; a.ld_qkv = ld;
  a.out = out; a.ld_out = ldo;
  a.B = c->Bm; a.Nt = c->Nt; a.Ni = c->Ni; a.H = c->H; a.hd = c->hd;
  return attention(c->dt, a, c->st);
}

// Modulation rows of (step i, block l, stream s): [Bm, chunks*C] at `stride`.
struct Mod {
  const float* p;
  int stride;
  const float* chunk(int j, int C) const { return p + (size_t)j * C; }
};

Mod block_mod(featfix_ctx* c, int i, int l, int s) {
  const int rb = c->mod_row_override >= 0 ? c->mod_row_override : c->need_row[i];
  return {c->bmodtab + (size_t)rb * c->Bm * c->Nblk + c->moff[2 * l + s], (int)c->Nblk};
}

Mod final_mod(featfix_ctx* c, int i) { return {c->fmodtab + (size_t)i * c->Bm * 2 * c->C, 2 * c->C}; }

cudaError_t ln_mod(featfix_ctx* c, const void* x, void* out, long long rows, const Mod& m, int shift_chunk,
                   int scale_chunk, int seg_split, int rpb0, int rpb1) {
  KTimer tm(c, FEATFIX_KCLASS_OTHER, 0);
  return launch_ln_mod(c->dt, x, out, rows, c->C, m.chunk(shift_chunk, c->C), m.chunk(scale_chunk, c->C), m.stride,
                       seg_split, rpb0, rpb1, c->st);
}

bool ln_fused(const featfix_ctx* c) { return !c->lncd_off.empty(); }

// The layer after LayerNorm k (0 before qkv / linear1, 1 before fc1) of
// block l, stream s (0 image / only, 1 text) reads the scaled copy in xm:
// its epilogue corrects the accumulator with the row statistics at `stats`
// and step i's per-sample tables.  Rows map to samples by
// seg_split / rpb0 / rpb1 (as for a gate).
void ln_consume(featfix_ctx* c, EpiArgs& e, int i, int l, int s, int k, const float2* stats, int seg_split, int rpb0,
                int rpb1) {
  const int j = c->lnjob_at[4 * l + 2 * s + k];
  const int rb = c->mod_row_override >= 0 ? c->mod_row_override : c->need_row[i];
  const int n = c->lnjob_n[j];
  const float* base = c->lncd + c->lncd_off[j] + (size_t)rb * c->Bm * 2 * n;
  e.ln_in = stats;
  e.ln_slots = c->C / 32;
  e.ln_cols = c->C;
  e.ln_c = base;
  e.ln_d = base + n;
  e.ln_cd_stride = 2 * n;
  e.seg_split = seg_split;
  e.rpb0 = rpb0;
  e.rpb1 = rpb1;
}

// This layer's output is the input of a LayerNorm with the scale chunk
// `scale_chunk` of m: its epilogue also writes the scaled copy (ln_out, at
// the GEMM's rows of xm) and the row statistics (stats).  The caller sets
// the row-to-sample mapping (the gate's).
void ln_produce(featfix_ctx* c, EpiArgs& e, const Mod& m, int scale_chunk, void* ln_out, float2* stats) {
  e.ln_scale = m.chunk(scale_chunk, c->C);
  e.ln_stride = m.stride;
  e.ln_out = ln_out;
  e.ln_stats = stats;
  e.ln_slots = c->C / 32;
}

float2* ln_rows(featfix_ctx* c, long long row0) { return c->lnst + row0 * (c->C / 32); }

// Exact DiT block B_l (Eq. 1): u -> out, optional history increment out - u.
featfix_status block_dit(featfix_ctx* ctx, int i, int l, const void* u, void* out, void* hist) {
  const int C = ctx->C, M = ctx->M, es = ctx->es;
  const long long T = ctx->T;
  const int wb = 11 + 10 * l;
  const auto& W = ctx->w;
  const Mod m = block_mod(ctx, i, l, 0);
  const bool fz = ln_fused(ctx);
  EpiArgs eq = epi(ctx->qkv, 3 * C, W[wb + 3]);
  if (fz && ctx->ln_src[0])
    ln_consume(ctx, eq, i, l, 0, 0, ctx->lnst, 0, 1, ctx->Ni);
  else
    FF_CK(ln_mod(ctx, u, ctx->xm, T, m, 0, 1, 0, 1, ctx->Ni));
  ctx->ln_src[0] = false;
  FF_CK(dense(ctx, (int)T, 3 * C, C, ctx->xm, C, W[wb + 2], eq));
  FF_CK(run_attention(ctx, ctx->qkv, off(ctx->qkv, C, es), off(ctx->qkv, 2 * C, es), 3 * C, ctx->att, C));
  EpiArgs e = epi(ctx->u1, C, W[wb + 5]);
  e.gate = m.chunk(2, C); e.gate_stride = m.stride; e.rpb1 = ctx->Ni;
  e.resid = u; e.ld_resid = C;
  if (fz) ln_produce(ctx, e, m, 4, ctx->xm, ctx->lnst);
  FF_CK(dense(ctx, (int)T, C, C, ctx->att, C, W[wb + 4], e));
  EpiArgs e1 = epi(ctx->big, M, W[wb + 7]);
  e1.act = 1;
  if (fz)
    ln_consume(ctx, e1, i, l, 0, 1, ctx->lnst, 0, 1, ctx->Ni);
  else
    FF_CK(ln_mod(ctx, ctx->u1, ctx->xm, T, m, 3, 4, 0, 1, ctx->Ni));
  FF_CK(dense(ctx, (int)T, M, C, ctx->xm, C, W[wb + 6], e1));
  EpiArgs e2 = epi(out, C, W[wb + 9]);
  e2.gate = m.chunk(5, C); e2.gate_stride = m.stride; e2.rpb1 = ctx->Ni;
  e2.resid = ctx->u1; e2.ld_resid = C;
  if (hist) { e2.hist_base = u; e2.hist_out = hist; }
  const bool feed = fz && ctx->ln_next;
  if (feed) ln_produce(ctx, e2, block_mod(ctx, i, l + 1, 0), 1, ctx->xm, ctx->lnst);
  FF_CK(dense(ctx, (int)T, C, M, ctx->big, M, W[wb + 8], e2));
  ctx->ln_src[0] = feed;
  return FEATFIX_OK;
}

// Exact MMDiT two-stream block: per-stream modulation and projections,
// joint attention.  Text rows [0, Bm*Nt), image rows after; each layer runs
// both streams in one grouped launch (image rows as group 0, text as group 1).
featfix_status block_dual(featfix_ctx* ctx, int i, int l, const void* u, void* out, void* hist) {
  const int C = ctx->C, M = ctx->M, es = ctx->es;
  const int wb = 10 + 20 * l;
  const auto& W = ctx->w;
  const long long rt = (long long)ctx->Bm * ctx->Nt, ri = (long long)ctx->Bm * ctx->Ni;
  const Mod mi = block_mod(ctx, i, l, 0), mt = block_mod(ctx, i, l, 1);
  const int ti = (int)ri, tt = (int)rt;
  const bool fz = ln_fused(ctx);
  // per-stream views: s = 0 text, 1 image (fused-LayerNorm job stream: 1 text, 0 image)
  auto rows0 = [&](int s_) { return s_ == 0 ? 0LL : rt; };
  auto rpb = [&](int s_) { return s_ ? ctx->Ni : ctx->Nt; };
  auto job_s = [&](int s_) { return s_ ? 0 : 1; };
  bool fin[2];
  for (int s = 0; s < 2; ++s) {
    const long long rows = s == 0 ? rt : ri;
    fin[s] = fz && ctx->ln_src[job_s(s)];
    if (rows && !fin[s])
      FF_CK(ln_mod(ctx, coff(u, rows0(s) * C, es), off(ctx->xm, rows0(s) * C, es), rows, s ? mi : mt, 0, 1, 0, 1,
                   rpb(s)));
  }
  ctx->ln_src[0] = ctx->ln_src[1] = false;
  EpiArgs qi = epi(off(ctx->qkv, rt * 3 * C, es), 3 * C, W[wb + 5]);
  if (ctx->rope) {
    qi.rope = ctx->rope; qi.rope_row0 = 0; qi.rope_period = ctx->Ni; qi.rope_cols = 2 * C; qi.rope_hd = ctx->hd;
  }
  EpiArgs qt = epi(ctx->qkv, 3 * C, W[wb + 7]);
  if (fin[1]) ln_consume(ctx, qi, i, l, 0, 0, ln_rows(ctx, rt), 0, 1, ctx->Ni);
  if (fin[0]) ln_consume(ctx, qt, i, l, 1, 0, ln_rows(ctx, 0), 0, 1, ctx->Nt);
  FF_CK(dense2(ctx, ti, off(ctx->xm, rt * C, es), W[wb + 4], qi, tt, ctx->xm, W[wb + 6], qt, 3 * C, C, C));
  FF_CK(run_attention(ctx, ctx->qkv, off(ctx->qkv, C, es), off(ctx->qkv, 2 * C, es), 3 * C, ctx->att, C));
  EpiArgs pe[2];
  for (int s = 0; s < 2; ++s) {
    const Mod& m = s ? mi : mt;
    const int wp = s ? wb + 8 : wb + 10;
    pe[s] = epi(off(ctx->u1, rows0(s) * C, es), C, W[wp + 1]);
    pe[s].gate = m.chunk(2, C); pe[s].gate_stride = m.stride; pe[s].rpb1 = rpb(s);
    pe[s].resid = coff(u, rows0(s) * C, es); pe[s].ld_resid = C;
    if (fz) ln_produce(ctx, pe[s], m, 4, off(ctx->xm, rows0(s) * C, es), ln_rows(ctx, rows0(s)));
  }
  FF_CK(dense2(ctx, ti, off(ctx->att, rt * C, es), W[wb + 8], pe[1], tt, ctx->att, W[wb + 10], pe[0], C, C, C));
  if (!fz) {
    for (int s = 0; s < 2; ++s) {
      const long long rows = s == 0 ? rt : ri;
      if (rows)
        FF_CK(ln_mod(ctx, off(ctx->u1, rows0(s) * C, es), off(ctx->xm, rows0(s) * C, es), rows, s ? mi : mt, 3, 4, 0,
                     1, rpb(s)));
    }
  }
  // the next block's first LayerNorm (a dual block: per stream; a single
  // block: one modulation for both streams)
  const bool feed = fz && ctx->ln_next;
  const bool next_dual = l + 1 < ctx->d.n_dual;
  EpiArgs f1[2], f2[2];
  for (int s = 0; s < 2; ++s) {
    const Mod& m = s ? mi : mt;
    const int wf = s ? wb + 12 : wb + 16;
    f1[s] = epi(off(ctx->big, rows0(s) * M, es), M, W[wf + 1]);
    f1[s].act = 1;
    if (fz) ln_consume(ctx, f1[s], i, l, job_s(s), 1, ln_rows(ctx, rows0(s)), 0, 1, rpb(s));
    f2[s] = epi(off(out, rows0(s) * C, es), C, W[wf + 3]);
    f2[s].gate = m.chunk(5, C); f2[s].gate_stride = m.stride; f2[s].rpb1 = rpb(s);
    f2[s].resid = off(ctx->u1, rows0(s) * C, es); f2[s].ld_resid = C;
    if (hist) { f2[s].hist_base = coff(u, rows0(s) * C, es); f2[s].hist_out = off(hist, rows0(s) * C, es); }
    if (feed)
      ln_produce(ctx, f2[s], block_mod(ctx, i, l + 1, next_dual ? job_s(s) : 0), 1, off(ctx->xm, rows0(s) * C, es),
                 ln_rows(ctx, rows0(s)));
  }
  FF_CK(dense2(ctx, ti, off(ctx->xm, rt * C, es), W[wb + 12], f1[1], tt, ctx->xm, W[wb + 16], f1[0], M, C, C));
  FF_CK(dense2(ctx, ti, off(ctx->big, rt * M, es), W[wb + 14], f2[1], tt, ctx->big, W[wb + 18], f2[0], C, M, M));
  ctx->ln_src[0] = feed && ri > 0;
  ctx->ln_src[1] = feed && rt > 0;
  return FEATFIX_OK;
}

// Exact MMDiT single-stream block: linear1 -> [q k v | GELU(mlp)] (the MLP
// half written next to the attention output), joint attention, linear2.
featfix_status block_single(featfix_ctx* ctx, int i, int l, const void* u, void* out, void* hist) {
  const int C = ctx->C, M = ctx->M;
  const int j = l - ctx->d.n_dual;
  const int wb = 10 + 20 * ctx->d.n_dual + 6 * j;
  const auto& W = ctx->w;
  const long long T = ctx->T, rt = (long long)ctx->Bm * ctx->Nt;
  const Mod m = block_mod(ctx, i, l, 0);
  const int rpb0 = ctx->Nt > 0 ? ctx->Nt : 1;
  const bool fz = ln_fused(ctx);
  const bool fin = fz && ctx->ln_src[0] && (rt == 0 || ctx->ln_src[1]);
  if (!fin) FF_CK(ln_mod(ctx, u, ctx->xm, T, m, 0, 1, (int)rt, rpb0, ctx->Ni));
  ctx->ln_src[0] = ctx->ln_src[1] = false;
  EpiArgs e = epi(ctx->qkv, 3 * C, W[wb + 3]);
  e.split_col = 3 * C;
  e.out2 = off(ctx->big, C, ctx->es);
  e.ldo2 = C + M;
  e.act = 1; e.act_col0 = 3 * C;
  if (ctx->rope) {
    e.rope = ctx->rope; e.rope_row0 = (int)rt; e.rope_period = ctx->Ni; e.rope_cols = 2 * C; e.rope_hd = ctx->hd;
  }
  if (fin) ln_consume(ctx, e, i, l, 0, 0, ctx->lnst, (int)rt, rpb0, ctx->Ni);
  FF_CK(dense(ctx, (int)T, 3 * C + M, C, ctx->xm, C, W[wb + 2], e));
  FF_CK(run_attention(ctx, ctx->qkv, off(ctx->qkv, C, ctx->es), off(ctx->qkv, 2 * C, ctx->es), 3 * C, ctx->big,
                      C + M));
  EpiArgs e2 = epi(out, C, W[wb + 5]);
  e2.gate = m.chunk(2, C); e2.gate_stride = m.stride;
  e2.seg_split = (int)rt; e2.rpb0 = rpb0; e2.rpb1 = ctx->Ni;
  e2.resid = u; e2.ld_resid = C;
  if (hist) { e2.hist_base = u; e2.hist_out = hist; }
  const bool feed = fz && ctx->ln_next;
  if (feed) ln_produce(ctx, e2, block_mod(ctx, i, l + 1, 0), 1, ctx->xm, ctx->lnst);
  FF_CK(dense(ctx, (int)T, C, C + M, ctx->big, C + M, W[wb + 4], e2));
  ctx->ln_src[0] = ctx->ln_src[1] = feed;
  return FEATFIX_OK;
}

featfix_status exact_block(featfix_ctx* ctx, int i, int l, const void* u, void* out, void* hist) {
  if (ctx->d.arch == FEATFIX_ARCH_DIT) return block_dit(ctx, i, l, u, out, hist);
  if (l < ctx->d.n_dual) return block_dual(ctx, i, l, u, out, hist);
  return block_single(ctx, i, l, u, out, hist);
}

// Conditioning and every adaLN modulation vector of steps [lo, hi):
// c = MLP(sinusoid(t)) (+ label embedding), then SiLU(c) times the
// concatenated modulation weights of all blocks (one GEMM) and of the final
// layer (one GEMM).  Only c depends on the step, so a whole trajectory's
// modulations are two tensor-core GEMMs.
featfix_status compute_mods(featfix_ctx* ctx, const void* cond, int lo, int hi) {
  const int S = hi - lo, C = ctx->C, Bm = ctx->Bm, es = ctx->es;
  const auto& W = ctx->w;
  const bool dit = ctx->d.arch == FEATFIX_ARCH_DIT;
  const int wfin = dit ? 7 : 6;
  {
    KTimer tm(ctx, FEATFIX_KCLASS_OTHER, 0);
    FF_CK(launch_sinusoid_table(ctx->dt, ctx->d_times + lo, S, off(ctx->sin_tab, (long long)lo * 256, es), ctx->st));
  }
  EpiArgs e1 = epi(off(ctx->thid_tab, (long long)lo * C, es), C, W[1]);
  e1.act = 2;
  FF_CK(dense(ctx, S, C, 256, off(ctx->sin_tab, (long long)lo * 256, es), 256, W[0], e1));
  EpiArgs e2 = epi(ctx->temb_tab + (size_t)lo * C, C, W[3]);
  e2.out_f32 = 1;
  FF_CK(dense(ctx, S, C, C, off(ctx->thid_tab, (long long)lo * C, es), C, W[2], e2));
  // row block of the first step in range that has exact blocks, and how many do
  int rb0 = -1, nneed = 0;
  for (int i = lo; i < hi; ++i)
    if (ctx->need_row[i] >= 0) {
      if (rb0 < 0) rb0 = ctx->need_row[i];
      ++nneed;
    }
  const bool gather = S > 1;
  {
    KTimer tm(ctx, FEATFIX_KCLASS_OTHER, 0);
    FF_CK(launch_cond_table(ctx->dt, ctx->temb_tab + (size_t)lo * C, dit ? W[4] : nullptr,
                            dit ? (const int*)cond : nullptr, S, Bm, C, gather ? ctx->d_need + lo : nullptr,
                            off(ctx->cs_all, (long long)lo * Bm * C, es), ctx->cs_need, ctx->st));
  }
  EpiArgs ef = epi(ctx->fmodtab + (size_t)lo * Bm * 2 * C, 2 * C, W[wfin + 1]);
  ef.out_f32 = 1;
  FF_CK(dense(ctx, S * Bm, 2 * C, C, off(ctx->cs_all, (long long)lo * Bm * C, es), C, W[wfin], ef));
  if (nneed > 0) {
    const void* A = gather ? off(ctx->cs_need, (long long)rb0 * Bm * C, es) : off(ctx->cs_all, (long long)lo * Bm * C, es);
    EpiArgs eb = epi(ctx->bmodtab + (size_t)rb0 * Bm * ctx->Nblk, (int)ctx->Nblk, ctx->bmod);
    eb.out_f32 = 1;
    FF_CK(dense(ctx, nneed * Bm, (int)ctx->Nblk, C, A, C, ctx->wmod, eb));
    if (ln_fused(ctx)) {
      // fused-LayerNorm tables of these row blocks: for every LayerNorm job,
      // rows (1 + scale) and shift times the next layer's weight
      const int nr = nneed * Bm;
      {
        KTimer tm(ctx, FEATFIX_KCLASS_OTHER, 0);
        FF_CK(launch_ln_ab(ctx->dt, ctx->bmodtab + (size_t)rb0 * Bm * ctx->Nblk, ctx->Nblk, nr, C, ctx->d_lnjobs,
                           (int)ctx->lnjobs.size(), ctx->lnab, ctx->lnab_job, ctx->st));
      }
      for (size_t j = 0; j < ctx->lnjobs.size(); ++j) {
        const int n = ctx->lnjob_n[j];
        EpiArgs ec = epi_plain(ctx->lncd + ctx->lncd_off[j] + (size_t)rb0 * Bm * 2 * n, n);
        ec.out_f32 = 1;
        FF_CK(dense(ctx, 2 * nr, n, C, off(ctx->lnab, (long long)j * ctx->lnab_job, es), C, ctx->lnjob_w[j], ec));
      }
    }
  }
  return FEATFIX_OK;
}

// Block-0 input: DiT patch embedding + position; MMDiT [text ; patches].
// feed: block 0 runs exact on this input, so the image rows' GEMM also
// writes the scaled copy and statistics of block 0's first LayerNorm.
featfix_status embed(featfix_ctx* ctx, int i, const float* latent, const void* cond, void* x, bool feed) {
  const auto& d = ctx->d;
  const int C = ctx->C, es = ctx->es;
  const long long rt = (long long)ctx->Bm * ctx->Nt;
  feed = feed && ln_fused(ctx);
  ctx->ln_src[0] = ctx->ln_src[1] = false;
  {
    KTimer tm(ctx, FEATFIX_KCLASS_OTHER, 0);
    FF_CK(launch_patchify(ctx->dt, latent, d.batch, ctx->Bm, d.in_ch, d.lat_f, d.lat_h, d.lat_w, d.patch, d.patch_t,
                          ctx->patches, ctx->st));
  }
  if (d.arch == FEATFIX_ARCH_DIT) {
    EpiArgs e = epi(x, C, ctx->w[6]);
    e.resid = ctx->pos; e.ld_resid = C;
    e.rpb1 = ctx->Ni;
    if (feed) ln_produce(ctx, e, block_mod(ctx, i, 0, 0), 1, ctx->xm, ctx->lnst);
    FF_CK(dense(ctx, ctx->Bm * ctx->Ni, C, ctx->fin, ctx->patches, ctx->fin, ctx->w[5], e));
  } else {
    if (rt) {
      KTimer tm(ctx, FEATFIX_KCLASS_OTHER, 0);
      FF_CK(launch_convert(ctx->dt, (const float*)cond, x, rt * C, ctx->st));
    }
    EpiArgs e = epi(off(x, rt * C, es), C, ctx->w[5]);
    e.rpb1 = ctx->Ni;
    if (feed) ln_produce(ctx, e, block_mod(ctx, i, 0, 0), 1, off(ctx->xm, rt * C, es), ln_rows(ctx, rt));
    FF_CK(dense(ctx, ctx->Bm * ctx->Ni, C, ctx->fin, ctx->patches, ctx->fin, ctx->w[4], e));
  }
  ctx->ln_src[0] = feed;
  return FEATFIX_OK;
}

// Final layer on the image rows and the guided sampler update.
featfix_status finish_step(featfix_ctx* ctx, int i, const void* x, float* latent) {
  const auto& d = ctx->d;
  const int C = ctx->C, es = ctx->es;
  const int wm = d.arch == FEATFIX_ARCH_DIT ? 7 : 6;
  const long long rt = (long long)ctx->Bm * ctx->Nt, ri = (long long)ctx->Bm * ctx->Ni;
  const Mod m = final_mod(ctx, i);
  FF_CK(ln_mod(ctx, coff(x, rt * C, es), ctx->xm, ri, m, 0, 1, 0, 1, ctx->Ni));
  EpiArgs e = epi(ctx->mout, ctx->fout, ctx->w[wm + 3]);
  e.out_f32 = 1;
  FF_CK(dense(ctx, (int)ri, ctx->fout, C, ctx->xm, C, ctx->w[wm + 2], e));
  float c1, c2;
  sampler_coeffs(ctx, i, &c1, &c2);
  KTimer tm(ctx, FEATFIX_KCLASS_OTHER, 0);
  FF_CK(launch_sampler(ctx->mout, latent, d.batch, d.cfg, d.cfg_scale, d.in_ch, d.out_ch, d.lat_f, d.lat_h, d.lat_w,
                       d.patch, d.patch_t, c1, c2, ctx->st));
  return FEATFIX_OK;
}

unsigned int* verify_counter(featfix_ctx* c) {
  return reinterpret_cast<unsigned int*>(reinterpret_cast<char*>(c->vws) + c->vws_bytes - 256);
}

void* ring_slot(featfix_ctx* c, int l, int slot) {
  return off(c->ring, ((long long)l * c->S + slot) * c->E, c->es);
}

Hist4 hist_ptrs(featfix_ctx* c, int l, int nt) {
  Hist4 h = {{nullptr, nullptr, nullptr, nullptr}};
  const int hd = c->bhead[l];
  for (int j = 0; j < nt; ++j) h.p[j] = ring_slot(c, l, ((hd - j) % c->S + c->S) % c->S);
  return h;
}

Hist4 sum_ptrs(featfix_ctx* c, int nt) {
  Hist4 h = {{nullptr, nullptr, nullptr, nullptr}};
  for (int j = 0; j < nt; ++j) h.p[j] = off(c->sring, (long long)(((c->head - j) % c->S + c->S) % c->S) * c->E, c->es);
  return h;
}

// Paid check of a site in the Verify arm on a shadow copy of the step's
// block-0 input: the per-block drafts chained up to each site, the exact
// block from the same incoming state (Eq. 3), the logged discrepancy (Eq. 4),
// then the draft continues (Verify forwards h_d).
featfix_status verify_shadow(featfix_ctx* ctx, int i, int nt, const float* wf) {
  const int L = ctx->L;
  int last = -1;
  for (int l = 0; l < L; ++l)
    if (ctx->kinds[(size_t)i * L + l] == FEATFIX_PLAN_SITE) last = l;
  if (last < 0) return FEATFIX_OK;
  const size_t bytes = (size_t)ctx->E * ctx->es;
  FF_CK(cudaMemcpyAsync(ctx->shadow, ctx->x0buf, bytes, cudaMemcpyDeviceToDevice, ctx->st));
  for (int l = 0; l <= last; ++l) {
    if (ctx->kinds[(size_t)i * L + l] == FEATFIX_PLAN_SITE) {
      ctx->ln_src[0] = ctx->ln_src[1] = false;
      FF_TRY(exact_block(ctx, i, l, ctx->shadow, ctx->xa, nullptr));
      ctx->cnt.paid_checks++;
      const int slot = (int)ctx->log_sites.size();
      if (slot >= ctx->max_logs) return fail(ctx, FEATFIX_ERR_STATE, "log overflow");
      KTimer tm(ctx, FEATFIX_KCLASS_VERIFY, (double)(nt + 3) * bytes);
      FF_CK(launch_verify(ctx->dt, ctx->shadow, hist_ptrs(ctx, l, nt), wf, nt, ctx->xa, ctx->E, 1,
                          ctx->dsums + 4 * slot, ctx->vws, ctx->st, nullptr, verify_counter(ctx)));
      ctx->log_sites.push_back({i, l});
    } else {
      // the run of drafted blocks up to the next site in one pass, as the
      // FeatFix arm's site steps do (so both arms reach their first site
      // with the same state)
      int l2 = l + 1;
      while (l2 <= last && l2 - l < SEG_MAX && ctx->kinds[(size_t)i * L + l2] == FEATFIX_PLAN_DRAFT) ++l2;
      if (l2 - l > 1) {
        HistSeg hs = {};
        for (int b = l; b < l2; ++b) {
          const Hist4 hp = hist_ptrs(ctx, b, nt);
          for (int j = 0; j < 4; ++j) hs.p[b - l][j] = hp.p[j];
        }
        KTimer tm(ctx, FEATFIX_KCLASS_DRAFT, (double)(nt * (l2 - l) + 2) * bytes);
        FF_CK(launch_draft_seg(ctx->dt, ctx->shadow, hs, l2 - l, wf, nt, ctx->E, ctx->st));
        l = l2 - 1;
        continue;
      }
      KTimer tm(ctx, FEATFIX_KCLASS_DRAFT, (double)(nt + 2) * bytes);
      FF_CK(launch_draft(ctx->dt, ctx->shadow, hist_ptrs(ctx, l, nt), wf, nt, ctx->E, ctx->st));
    }
  }
  return FEATFIX_OK;
}

// One denoising step (modulations of step i ready): embedding, the L blocks
// per the plan (exact / draft / paid site), final layer, sampler update.
featfix_status step_body(featfix_ctx* ctx, float* latent, int i, const void* cond) {
  if (i == 0) {
    ctx->head = ctx->S - 1;
    ctx->bhead.assign(ctx->L, ctx->S - 1);
    ctx->count = 0;
    ctx->cnt = {0, 0, 0, 0};
    ctx->log_sites.clear();
  }
  const int L = ctx->L;
  const bool refresh = ctx->isref[i] != 0;
  const bool vanilla = ctx->mode == FEATFIX_MODE_VANILLA;
  const size_t bytes = (size_t)ctx->E * ctx->es;
  // all blocks exact and chained (full refresh, vanilla): each block's
  // output GEMM also prepares the next block's first LayerNorm
  const bool chain = refresh || vanilla;
  FF_TRY(embed(ctx, i, latent, cond, ctx->x0buf, chain && ctx->kinds[(size_t)i * L] == FEATFIX_PLAN_EXACT));
  const int new_slot = (ctx->head + 1) % ctx->S;
  const bool site_push = (ctx->flags & FEATFIX_FLAG_SITE_UPDATES_HISTORY) != 0;
  int nt = ctx->keff[i] + 1;
  float wf[4];
  for (int j = 0; j < 4; ++j) wf[j] = (float)ctx->wts[(size_t)i * 4 + j];
  // block l's draft order and weights (its own history when sites push)
  auto block_weights = [&](int l) {
    if (!site_push) return;
    nt = ctx->keff_bl[(size_t)i * L + l] + 1;
    for (int j = 0; j < 4; ++j) wf[j] = (float)ctx->wts_bl[((size_t)i * L + l) * 4 + j];
  };
  bool has_site = false, has_capture = false;
  for (int l = 0; l < L; ++l) has_site |= ctx->kinds[(size_t)i * L + l] == FEATFIX_PLAN_SITE;
  for (auto& cp : ctx->caps) has_capture |= cp.step == i;
  const bool telescope = !refresh && !vanilla && !has_capture && !site_push &&
                         !(ctx->flags & FEATFIX_FLAG_PER_BLOCK_DRAFT) && (!has_site || ctx->mode == FEATFIX_MODE_VERIFY);
  // drafted blocks between the sites of a per-block step: one pass per run
  const bool seg_ok = !site_push && !has_capture && !(ctx->flags & FEATFIX_FLAG_PER_BLOCK_DRAFT);
  void* x = ctx->x0buf;
  if (telescope) {
    if (has_site) FF_TRY(verify_shadow(ctx, i, nt, wf));
    KTimer tm(ctx, FEATFIX_KCLASS_DRAFT, (double)(nt + 2) * bytes);
    FF_CK(launch_draft(ctx->dt, x, sum_ptrs(ctx, nt), wf, nt, ctx->E, ctx->st));
  } else {
    // x0buf, then ping-pong xa / xb: x0buf stays the step's input for the
    // refresh sum below
    void* y = ctx->xa;
    auto advance = [&]() {  // the block wrote y: it becomes the state
      x = y;
      y = (x == ctx->xa) ? ctx->xb : ctx->xa;
    };
    for (int l = 0; l < L; ++l) {
      const unsigned char kind = ctx->kinds[(size_t)i * L + l];
      for (auto& cp : ctx->caps) {
        if (cp.step != i || cp.layer != l) continue;
        if (cp.in) FF_CK(cudaMemcpyAsync(cp.in, x, bytes, cudaMemcpyDeviceToDevice, ctx->st));
        if (cp.nhist > 0 && kind != FEATFIX_PLAN_EXACT) {
          block_weights(l);
          const Hist4 hp = hist_ptrs(ctx, l, nt);
          for (int j = 0; j < std::min(cp.nhist, nt); ++j)
            FF_CK(cudaMemcpyAsync(cp.hist[j], hp.p[j], bytes, cudaMemcpyDeviceToDevice, ctx->st));
        }
      }
      const int bslot = (ctx->bhead[l] + 1) % ctx->S;  // block l's next ring slot
      if (kind == FEATFIX_PLAN_EXACT) {
        void* hist = (refresh && !vanilla) ? ring_slot(ctx, l, bslot) : nullptr;
        ctx->ln_next = chain && l + 1 < L;
        FF_TRY(exact_block(ctx, i, l, x, y, hist));
        ctx->ln_next = false;
        advance();
      } else if (kind == FEATFIX_PLAN_DRAFT) {
        block_weights(l);
        // a run of drafted blocks in one pass (same weights for every block;
        // per block with site pushes, captures or FEATFIX_FLAG_PER_BLOCK_DRAFT)
        int l2 = l + 1;
        if (seg_ok)
          while (l2 < L && l2 - l < SEG_MAX && ctx->kinds[(size_t)i * L + l2] == FEATFIX_PLAN_DRAFT) ++l2;
        if (l2 - l > 1) {
          HistSeg hs = {};
          for (int b = l; b < l2; ++b) {
            const Hist4 hp = hist_ptrs(ctx, b, nt);
            for (int j = 0; j < 4; ++j) hs.p[b - l][j] = hp.p[j];
          }
          KTimer tm(ctx, FEATFIX_KCLASS_DRAFT, (double)(nt * (l2 - l) + 2) * bytes);
          FF_CK(launch_draft_seg(ctx->dt, x, hs, l2 - l, wf, nt, ctx->E, ctx->st));
          l = l2 - 1;
          continue;
        }
        KTimer tm(ctx, FEATFIX_KCLASS_DRAFT, (double)(nt + 2) * bytes);
        FF_CK(launch_draft(ctx->dt, x, hist_ptrs(ctx, l, nt), wf, nt, ctx->E, ctx->st));
      } else {
        block_weights(l);
        // with site pushes the exact increment goes to the spare slot; the
        // draft below still reads the K_eff + 1 entries before it
        ctx->ln_src[0] = ctx->ln_src[1] = false;  // the input comes from a draft
        FF_TRY(exact_block(ctx, i, l, x, y, site_push ? ring_slot(ctx, l, bslot) : nullptr));
        ctx->cnt.paid_checks++;
        if (ctx->mode != FEATFIX_MODE_EXACT_ONLY) {
          const int slot = (int)ctx->log_sites.size();
          if (slot >= ctx->max_logs) return fail(ctx, FEATFIX_ERR_STATE, "log overflow");
          const int wr = ctx->mode == FEATFIX_MODE_VERIFY ? 1 : 0;
          // partial forwarding arm: h_f only on the selected tokens / channels
          const bool partial = ctx->mode == FEATFIX_MODE_FEATFIX && ctx->fmask_axis != FEATFIX_MASK_NONE;
          const FwdMix fm = {y, ctx->fmask_axis == FEATFIX_MASK_TOKENS ? ctx->d_rmask : nullptr,
                             ctx->fmask_axis == FEATFIX_MASK_CHANNELS ? ctx->d_cmask : nullptr, ctx->C};
          KTimer tm(ctx, FEATFIX_KCLASS_VERIFY, (double)(nt + 2 + wr + (partial ? 1 : 0)) * bytes);
          FF_CK(launch_verify(ctx->dt, x, hist_ptrs(ctx, l, nt), wf, nt, y, ctx->E, wr, ctx->dsums + 4 * slot,
                              ctx->vws, ctx->st, partial ? &fm : nullptr, verify_counter(ctx)));
          ctx->log_sites.push_back({i, l});
        }
        if (ctx->mode != FEATFIX_MODE_VERIFY) {
          advance();
          ctx->cnt.forwarded++;
        }
        if (site_push) ctx->bhead[l] = bslot;
      }
      for (auto& cp : ctx->caps)
        if (cp.step == i && cp.layer == l && cp.out) FF_CK(cudaMemcpyAsync(cp.out, x, bytes, cudaMemcpyDeviceToDevice, ctx->st));
    }
  }
  if (refresh && !vanilla) {
    KTimer tm(ctx, FEATFIX_KCLASS_OTHER, 0);
    FF_CK(launch_diff(ctx->dt, x, ctx->x0buf, off(ctx->sring, (long long)new_slot * ctx->E, ctx->es), ctx->E, ctx->st));
    ctx->head = new_slot;
    for (int l = 0; l < L; ++l) ctx->bhead[l] = (ctx->bhead[l] + 1) % ctx->S;
    ctx->count = std::min(ctx->count + 1, ctx->S);
  }
  if (refresh || vanilla) ctx->cnt.refresh_steps++;
  FF_TRY(finish_step(ctx, i, x, latent));
  ctx->cnt.steps_done = i + 1;
  ctx->next_step = i + 1;
  return FEATFIX_OK;
}

// The whole trajectory on the fixed input buffers g_lat / g_cond.
featfix_status trajectory(featfix_ctx* ctx) {
  FF_TRY(compute_mods(ctx, ctx->g_cond, 0, ctx->steps));
  for (int i = 0; i < ctx->steps; ++i) FF_TRY(step_body(ctx, ctx->g_lat, i, ctx->g_cond));
  return FEATFIX_OK;
}

// Capture trajectory() into a graph on the private stream.  The host-side
// trajectory state (history ring position, counters, log slots) advances
// during the capture exactly as in a run from step 0, and every replay
// repeats that run, so the state stays valid after each replay.
featfix_status build_graph(featfix_ctx* ctx) {
  graph_reset(ctx);
  FF_CK(cudaStreamBeginCapture(ctx->cap_st, cudaStreamCaptureModeRelaxed));
  ctx->st = ctx->cap_st;
  ctx->capturing = true;
  const long long k0 = launches_total();
  const featfix_status s = trajectory(ctx);
  ctx->capturing = false;
  ctx->st = ctx->user_st;
  cudaGraph_t g = nullptr;
  const cudaError_t e = cudaStreamEndCapture(ctx->cap_st, &g);
  ctx->graph_kernels = launches_total() - k0;
  count_launches(-ctx->graph_kernels);  // capturing launched nothing; replays are counted
  if (s != FEATFIX_OK) {
    if (g) cudaGraphDestroy(g);
    graph_reset(ctx);
    return s;
  }
  if (e != cudaSuccess) return fail(ctx, FEATFIX_ERR_CUDA, std::string("graph capture: ") + cudaGetErrorString(e));
  const cudaError_t e2 = cudaGraphInstantiate(&ctx->gexec, g, 0);
  cudaGraphDestroy(g);
  if (e2 != cudaSuccess) {
    ctx->gexec = nullptr;
    return fail(ctx, FEATFIX_ERR_CUDA, std::string("graph instantiate: ") + cudaGetErrorString(e2));
  }
  ctx->graph_ok = true;
  return FEATFIX_OK;
}

void free_all(featfix_ctx* c) {
  graph_reset(c);
  void* bufs[] = {c->xa, c->xb, c->xm, c->qkv, c->att, c->u1, c->big, c->patches, c->pos, c->mout, c->rope,
                  c->ring, c->sring, c->x0buf, c->shadow, c->wmod, c->bmod, c->d_times, c->d_need, c->sin_tab, c->thid_tab, c->temb_tab,
                  c->cs_all, c->cs_need, c->bmodtab, c->fmodtab, c->dsums, c->vws, c->g_lat, c->g_cond,
                  c->h_latent, c->h_cond, c->d_rmask, c->d_cmask, c->lnst, c->lncd, c->lnab, c->d_lnjobs};
  for (void* p : bufs)
    if (p) cudaFree(p);
  for (int k = 0; k < NKCLASS; ++k)
    for (auto& t : c->pending[k]) { cudaEventDestroy(t.a); cudaEventDestroy(t.b); }
  for (auto e : c->evpool) cudaEventDestroy(e);
  if (c->cap_st) cudaStreamDestroy(c->cap_st);
}

featfix_status alloc(featfix_ctx* c, void** p, size_t bytes) {
  if (cudaMalloc(p, bytes ? bytes : 16) != cudaSuccess) {
    cudaGetLastError();
    *p = nullptr;
    return fail(c, FEATFIX_ERR_OOM, "device allocation of " + std::to_string(bytes) + " bytes failed");
  }
  return FEATFIX_OK;
}

void free_ptr(void** p) {
  if (*p) cudaFree(*p);
  *p = nullptr;
}

// (cos, sin) of every image token / rotary pair: axis widths d/2,d/2 (2-D)
// or d/8, 7d/16, 7d/16 (3-D); pair j of an axis of width w turns by
// pos * 10000^(-2j/w).
std::vector<float2> rope_table_host(const featfix_model_desc& d, int hd) {
  std::vector<int> axes;
  if (d.rope_dims == 2) axes = {hd / 2, hd / 2};
  else {
    const int t = hd / 8, hw = (hd - t) / 2;
    axes = {t, hw, hd - t - hw};
  }
  const int gf = d.lat_f > 0 ? d.lat_f / d.patch_t : 1, gh = d.lat_h / d.patch, gw = d.lat_w / d.patch;
  const int ni = gf * gh * gw;
  std::vector<float2> tab((size_t)ni * (hd / 2));
  for (int n = 0; n < ni; ++n) {
    int pos[3];
    if (d.rope_dims == 2) { pos[0] = (n / gw) % gh; pos[1] = n % gw; }
    else { pos[0] = n / (gw * gh); pos[1] = (n / gw) % gh; pos[2] = n % gw; }
    int col = 0;
    for (size_t a = 0; a < axes.size(); ++a) {
      for (int j = 0; j < axes[a] / 2; ++j, ++col) {
        const double ang = pos[a] * std::pow(10000.0, -2.0 * j / axes[a]);
        tab[(size_t)n * (hd / 2) + col] = make_float2((float)std::cos(ang), (float)std::sin(ang));
      }
    }
  }
  return tab;
}

// Block modulation weights gathered into one [Nblk, C] matrix (and bias);
// the caller's tensors are copied once here.
featfix_status gather_mod_weights(featfix_ctx* ctx) {
  const auto& d = ctx->d;
  const int C = ctx->C, es = ctx->es;
  std::vector<std::pair<int, int>> parts;  // (weight index, rows)
  ctx->moff.assign(2 * (size_t)ctx->L, 0);
  long long col = 0;
  for (int l = 0; l < ctx->L; ++l) {
    if (d.arch == FEATFIX_ARCH_DIT) {
      ctx->moff[2 * l] = col;
      parts.push_back({11 + 10 * l, 6 * C});
      col += 6 * C;
    } else if (l < d.n_dual) {
      ctx->moff[2 * l] = col;
      parts.push_back({10 + 20 * l, 6 * C});
      col += 6 * C;
      ctx->moff[2 * l + 1] = col;
      parts.push_back({10 + 20 * l + 2, 6 * C});
      col += 6 * C;
    } else {
      ctx->moff[2 * l] = col;
      parts.push_back({10 + 20 * d.n_dual + 6 * (l - d.n_dual), 3 * C});
      col += 3 * C;
    }
  }
  ctx->Nblk = col;
  FF_TRY(alloc(ctx, &ctx->wmod, (size_t)col * C * es));
  FF_TRY(alloc(ctx, &ctx->bmod, (size_t)col * es));
  long long r = 0;
  for (auto& p : parts) {
    FF_CK(cudaMemcpyAsync(off(ctx->wmod, r * C, es), ctx->w[p.first], (size_t)p.second * C * es,
                          cudaMemcpyDeviceToDevice, ctx->user_st));
    FF_CK(cudaMemcpyAsync(off(ctx->bmod, r, es), ctx->w[p.first + 1], (size_t)p.second * es,
                          cudaMemcpyDeviceToDevice, ctx->user_st));
    r += p.second;
  }
  return FEATFIX_OK;
}

// Jobs of the fused LayerNorm: every adaLN LayerNorm whose next layer is a
// tensor-core GEMM -- DiT and dual blocks: before qkv (shift/scale chunks
// 0/1) and before fc1 (3/4) per stream; single blocks: before linear1 (0/1).
featfix_status setup_ln_jobs(featfix_ctx* ctx) {
  const auto& d = ctx->d;
  const long long C = ctx->C, M = ctx->M;
  ctx->lnf = ctx->dt == BF16 && C % 64 == 0;   // an even number of 32-column chunks per row
  ctx->lnjob_at.assign(4 * (size_t)ctx->L, -1);
  if (!ctx->lnf) return FEATFIX_OK;
  auto add = [&](int l, int s, int k, int w, long long n) {
    const long long col = ctx->moff[2 * l + s];
    const int shc = k == 0 ? 0 : 3, scc = k == 0 ? 1 : 4;
    ctx->lnjob_at[4 * l + 2 * s + k] = (int)ctx->lnjobs.size();
    ctx->lnjobs.push_back(make_int2((int)(col + scc * C), (int)(col + shc * C)));
    ctx->lnjob_n.push_back((int)n);
    ctx->lnjob_w.push_back(ctx->w[w]);
  };
  for (int l = 0; l < ctx->L; ++l) {
    if (d.arch == FEATFIX_ARCH_DIT) {
      const int wb = 11 + 10 * l;
      add(l, 0, 0, wb + 2, 3 * C);
      add(l, 0, 1, wb + 6, M);
    } else if (l < d.n_dual) {
      const int wb = 10 + 20 * l;
      add(l, 0, 0, wb + 4, 3 * C);
      add(l, 0, 1, wb + 12, M);
      add(l, 1, 0, wb + 6, 3 * C);
      add(l, 1, 1, wb + 16, M);
    } else {
      const int wb = 10 + 20 * d.n_dual + 6 * (l - d.n_dual);
      add(l, 0, 0, wb + 2, 3 * C + M);
    }
  }
  FF_TRY(alloc(ctx, (void**)&ctx->lnst, (size_t)ctx->T * (C / 32) * sizeof(float2)));
  FF_TRY(alloc(ctx, (void**)&ctx->d_lnjobs, ctx->lnjobs.size() * sizeof(int2)));
  FF_CK(cudaMemcpy(ctx->d_lnjobs, ctx->lnjobs.data(), ctx->lnjobs.size() * sizeof(int2), cudaMemcpyHostToDevice));
  return FEATFIX_OK;
}

featfix_status create_impl(featfix_ctx* ctx) {
  const featfix_model_desc& d = ctx->d;
  const int es = ctx->es;
  const long long T = ctx->T, C = ctx->C, M = ctx->M;
  FF_CK(cudaStreamCreateWithFlags(&ctx->cap_st, cudaStreamNonBlocking));
  FF_TRY(alloc(ctx, &ctx->xa, T * C * es));
  FF_TRY(alloc(ctx, &ctx->xb, T * C * es));
  FF_TRY(alloc(ctx, &ctx->x0buf, T * C * es));
  FF_TRY(alloc(ctx, &ctx->shadow, T * C * es));
  FF_TRY(alloc(ctx, &ctx->xm, T * C * es));
  FF_TRY(alloc(ctx, &ctx->qkv, T * 3 * C * es));
  FF_TRY(alloc(ctx, &ctx->att, T * C * es));
  FF_TRY(alloc(ctx, &ctx->u1, T * C * es));
  FF_TRY(alloc(ctx, &ctx->big, T * (C + M) * es));
  FF_TRY(alloc(ctx, &ctx->patches, (size_t)ctx->Bm * ctx->Ni * ctx->fin * es));
  FF_TRY(alloc(ctx, (void**)&ctx->mout, (size_t)ctx->Bm * ctx->Ni * ctx->fout * 4));
  ctx->lat_elems = (long long)d.batch * d.in_ch * (d.lat_f > 0 ? d.lat_f : 1) * d.lat_h * d.lat_w;
  ctx->cond_bytes = d.arch == FEATFIX_ARCH_DIT ? (size_t)ctx->Bm * sizeof(int)
                                              : (size_t)ctx->Bm * ctx->Nt * ctx->C * sizeof(float);
  FF_TRY(alloc(ctx, (void**)&ctx->g_lat, (size_t)ctx->lat_elems * 4));
  FF_TRY(alloc(ctx, &ctx->g_cond, ctx->cond_bytes));
  if (d.arch == FEATFIX_ARCH_DIT) {
    FF_TRY(alloc(ctx, &ctx->pos, (size_t)ctx->Bm * ctx->Ni * C * es));
    FF_CK(launch_pos2d(ctx->dt, ctx->pos, ctx->Bm, ctx->gh, ctx->gw, ctx->C, ctx->user_st));
  }
  if (d.arch == FEATFIX_ARCH_MMDIT && d.rope_dims) {
    FF_TRY(alloc(ctx, (void**)&ctx->rope, (size_t)ctx->Ni * (ctx->hd / 2) * sizeof(float2)));
    std::vector<float2> tab = rope_table_host(d, ctx->hd);
    FF_CK(cudaMemcpyAsync(ctx->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice, ctx->user_st));
    FF_CK(cudaStreamSynchronize(ctx->user_st));
  }
  FF_TRY(gather_mod_weights(ctx));
  FF_TRY(setup_ln_jobs(ctx));
  FF_CK(cudaStreamSynchronize(ctx->user_st));
  return FEATFIX_OK;
}

// Per-schedule device state: history ring, modulation tables, logs.
featfix_status schedule_buffers(featfix_ctx* ctx, int steps, int K, int mode, int n_sites, unsigned flags) {
  const int es = ctx->es, C = ctx->C, Bm = ctx->Bm;
  // K + 1 increments per block; a site that pushes its increment writes a
  // slot while its own draft still reads the K + 1 newest: one spare slot
  const int S = K + 1 + ((flags & FEATFIX_FLAG_SITE_UPDATES_HISTORY) ? 1 : 0);
  if (ctx->ring && ctx->S != S) {
    free_ptr(&ctx->ring);
    free_ptr(&ctx->sring);
  }
  if (!ctx->ring && mode != FEATFIX_MODE_VANILLA) {
    FF_TRY(alloc(ctx, &ctx->ring, (size_t)ctx->L * S * ctx->E * es));
    FF_TRY(alloc(ctx, &ctx->sring, (size_t)S * ctx->E * es));
  }
  ctx->S = S;
  const int nlog = std::max(n_sites, 1);
  if (nlog > ctx->max_logs) {
    free_ptr((void**)&ctx->dsums);
    FF_TRY(alloc(ctx, (void**)&ctx->dsums, (size_t)nlog * 4 * sizeof(double)));
    ctx->max_logs = nlog;
  }
  // the partials, then the completion counter of the one-launch reduction
  verify_prepare();  // host-side occupancy query, kept out of the graph capture
  const size_t need = (verify_workspace_bytes(ctx->E) + 255) / 256 * 256 + 256;
  if (need > ctx->vws_bytes) {
    free_ptr(&ctx->vws);
    FF_TRY(alloc(ctx, &ctx->vws, need));
    FF_CK(cudaMemsetAsync(ctx->vws, 0, need, ctx->user_st));
    ctx->vws_bytes = need;
  }
  void** tabs[] = {(void**)&ctx->d_times, (void**)&ctx->d_need, &ctx->sin_tab, &ctx->thid_tab, (void**)&ctx->temb_tab,
                   &ctx->cs_all, &ctx->cs_need, (void**)&ctx->bmodtab, (void**)&ctx->fmodtab};
  for (void** p : tabs) free_ptr(p);
  const int nn = std::max(ctx->n_need, 1);
  FF_TRY(alloc(ctx, (void**)&ctx->d_times, (size_t)steps * 4));
  FF_TRY(alloc(ctx, (void**)&ctx->d_need, (size_t)steps * 4));
  FF_TRY(alloc(ctx, &ctx->sin_tab, (size_t)steps * 256 * es));
  FF_TRY(alloc(ctx, &ctx->thid_tab, (size_t)steps * C * es));
  FF_TRY(alloc(ctx, (void**)&ctx->temb_tab, (size_t)steps * C * 4));
  FF_TRY(alloc(ctx, &ctx->cs_all, (size_t)steps * Bm * C * es));
  FF_TRY(alloc(ctx, &ctx->cs_need, (size_t)nn * Bm * C * es));
  FF_TRY(alloc(ctx, (void**)&ctx->bmodtab, (size_t)(nn + 1) * Bm * ctx->Nblk * 4));
  FF_TRY(alloc(ctx, (void**)&ctx->fmodtab, (size_t)steps * Bm * 2 * C * 4));
  // fused-LayerNorm tables: one row block per modulation row block
  free_ptr((void**)&ctx->lncd);
  free_ptr(&ctx->lnab);
  ctx->lncd_off.clear();
  if (ctx->lnf && (flags & FEATFIX_FLAG_FUSED_LN)) {
    const long long rows = (long long)(nn + 1) * Bm;
    long long tot = 0;
    for (int n : ctx->lnjob_n) {
      ctx->lncd_off.push_back(tot);
      tot += 2 * rows * n;
    }
    ctx->ln_rb = nn + 1;
    ctx->lnab_job = 2 * rows * C;
    FF_TRY(alloc(ctx, (void**)&ctx->lncd, (size_t)tot * 4));
    FF_TRY(alloc(ctx, &ctx->lnab, (size_t)ctx->lnjobs.size() * ctx->lnab_job * es));
  }
  return FEATFIX_OK;
}

}  // namespace

// ============================================================================
// C ABI
// ============================================================================
extern "C" {

const char* featfix_status_string(featfix_status s) {
  switch (s) {
    case FEATFIX_OK: return "ok";
    case FEATFIX_ERR_INVALID_ARG: return "invalid argument";
    case FEATFIX_ERR_SCHEDULE: return "schedule rule violated";
    case FEATFIX_ERR_STATE: return "call out of order";
    case FEATFIX_ERR_OOM: return "out of device memory";
    case FEATFIX_ERR_CUDA: return "CUDA error";
    case FEATFIX_ERR_UNSUPPORTED: return "unsupported";
  }
  return "unknown status";
}

long long featfix_launch_count(void) { return launches_total(); }

const char* featfix_last_error(const featfix_ctx* ctx) { return ctx ? ctx->err.c_str() : "null context"; }

int featfix_weight_count(const featfix_model_desc* d) {
  if (!check_desc(d).empty()) return -1;
  if (d->arch == FEATFIX_ARCH_DIT) return 11 + 10 * d->n_dual;
  return 10 + 20 * d->n_dual + 6 * d->n_single;
}

long long featfix_token_row(const featfix_model_desc* d, int b, int n) {
  if (!d) return -1;
  const int bm = d->batch * (d->cfg ? 2 : 1);
  const int nt = d->txt_tokens, ni = img_tokens(*d);
  if (b < 0 || b >= bm || n < 0 || n >= nt + ni) return -1;
  return n < nt ? (long long)b * nt + n : (long long)bm * nt + (long long)b * ni + (n - nt);
}

featfix_status featfix_plan_build(int steps, int n_layers_, const int* refresh, int n_refresh, int draft_order,
                                  const featfix_site* sites, int n_sites, int mode, unsigned flags,
                                  unsigned char* kinds, int* k_eff, double* weights) {
  std::vector<unsigned char> kd;
  std::vector<int> ke, keb;
  std::vector<double> wt, wtb;
  std::vector<char> isref;
  std::string err;
  featfix_status s = plan_core(steps, n_layers_, refresh, n_refresh, draft_order, sites, n_sites, mode, flags, kd, ke,
                               wt, isref, keb, wtb, err);
  if (s != FEATFIX_OK) return s;
  if (kinds) std::memcpy(kinds, kd.data(), kd.size());
  if (k_eff) std::memcpy(k_eff, ke.data(), ke.size() * sizeof(int));
  if (weights) std::memcpy(weights, wt.data(), wt.size() * sizeof(double));
  return FEATFIX_OK;
}

featfix_status featfix_plan_build_blocks(int steps, int n_layers_, const int* refresh, int n_refresh, int draft_order,
                                         const featfix_site* sites, int n_sites, int mode, unsigned flags, int* k_eff,
                                         double* weights) {
  std::vector<unsigned char> kd;
  std::vector<int> ke, keb;
  std::vector<double> wt, wtb;
  std::vector<char> isref;
  std::string err;
  featfix_status s = plan_core(steps, n_layers_, refresh, n_refresh, draft_order, sites, n_sites, mode, flags, kd, ke,
                               wt, isref, keb, wtb, err);
  if (s != FEATFIX_OK) return s;
  if (k_eff) std::memcpy(k_eff, keb.data(), keb.size() * sizeof(int));
  if (weights) std::memcpy(weights, wtb.data(), wtb.size() * sizeof(double));
  return FEATFIX_OK;
}

featfix_status featfix_create(const featfix_model_desc* desc, const void* const* dev_weights, int n_weights,
                              void* cuda_stream, featfix_ctx** out) {
  if (!out) return FEATFIX_ERR_INVALID_ARG;
  *out = nullptr;
  if (!check_desc(desc).empty()) return FEATFIX_ERR_INVALID_ARG;
  const int nw = featfix_weight_count(desc);
  if (!dev_weights || n_weights != nw) return FEATFIX_ERR_INVALID_ARG;
  for (int k = 0; k < nw; ++k)
    if (!dev_weights[k] || ((uintptr_t)dev_weights[k] & 15)) return FEATFIX_ERR_INVALID_ARG;

  featfix_ctx* ctx = new featfix_ctx();
  const featfix_model_desc& d = *desc;
  ctx->d = d;
  ctx->dt = d.dtype == FEATFIX_DTYPE_BF16 ? BF16 : F32;
  ctx->es = dsize(ctx->dt);
  ctx->L = n_layers(d);
  ctx->Bm = d.batch * (d.cfg ? 2 : 1);
  ctx->Nt = d.txt_tokens;
  ctx->Ni = img_tokens(d);
  ctx->Ntot = ctx->Nt + ctx->Ni;
  ctx->C = d.hidden;
  ctx->H = d.heads;
  ctx->hd = d.head_dim;
  ctx->M = d.mlp;
  ctx->P = patch_vol(d);
  ctx->fin = ctx->P * d.in_ch;
  ctx->fout = ctx->P * d.out_ch;
  ctx->T = (long long)ctx->Bm * ctx->Ntot;
  ctx->E = ctx->T * ctx->C;
  ctx->gf = d.lat_f > 0 ? d.lat_f / d.patch_t : 1;
  ctx->gh = d.lat_h / d.patch;
  ctx->gw = d.lat_w / d.patch;
  ctx->w.assign(dev_weights, dev_weights + nw);
  ctx->user_st = reinterpret_cast<cudaStream_t>(cuda_stream);
  ctx->st = ctx->user_st;
  const featfix_status s = create_impl(ctx);
  if (s != FEATFIX_OK) {
    free_all(ctx);
    delete ctx;
    return s;
  }
  *out = ctx;
  return FEATFIX_OK;
}

void featfix_destroy(featfix_ctx* ctx) {
  if (!ctx) return;
  cudaStreamSynchronize(ctx->user_st);
  free_all(ctx);
  delete ctx;
}

featfix_status featfix_set_schedule(featfix_ctx* ctx, int steps, const int* refresh, int n_refresh, int draft_order,
                                    const featfix_site* sites, int n_sites, int mode, unsigned flags) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  std::vector<unsigned char> kd;
  std::vector<int> ke, keb;
  std::vector<double> wt, wtb;
  std::vector<char> isref;
  std::string err;
  featfix_status s = plan_core(steps, ctx->L, refresh, n_refresh, draft_order, sites, n_sites, mode, flags, kd, ke, wt,
                               isref, keb, wtb, err);
  if (s != FEATFIX_OK) return fail(ctx, s, err);
  if (ctx->d.sampler == FEATFIX_SAMPLER_DDIM && (1000 % steps != 0))
    return fail(ctx, FEATFIX_ERR_UNSUPPORTED, "DDIM needs steps dividing 1000");
  FF_CK(cudaStreamSynchronize(ctx->user_st));
  graph_reset(ctx);
  ctx->sched = false;
  // steps whose blocks need modulation vectors (any exact block or site)
  std::vector<int> need(steps, -1);
  int nn = 0;
  for (int i = 0; i < steps; ++i) {
    bool any = false;
    for (int l = 0; l < ctx->L; ++l) any |= kd[(size_t)i * ctx->L + l] != FEATFIX_PLAN_DRAFT;
    if (any) need[i] = nn++;
  }
  ctx->n_need = nn;
  FF_TRY(schedule_buffers(ctx, steps, draft_order, mode, n_sites, flags));
  ctx->need_row = need;
  ctx->steps = steps;
  std::vector<float> times(steps);
  for (int i = 0; i < steps; ++i) times[i] = (float)model_time(ctx, i);
  FF_CK(cudaMemcpy(ctx->d_times, times.data(), steps * sizeof(float), cudaMemcpyHostToDevice));
  FF_CK(cudaMemcpy(ctx->d_need, need.data(), steps * sizeof(int), cudaMemcpyHostToDevice));
  ctx->kinds.swap(kd);
  ctx->keff.swap(ke);
  ctx->wts.swap(wt);
  ctx->keff_bl.swap(keb);
  ctx->wts_bl.swap(wtb);
  ctx->isref.swap(isref);
  ctx->K = draft_order;
  ctx->mode = mode;
  ctx->flags = flags;
  ctx->sched = true;
  ctx->next_step = 0;
  ctx->cnt = {0, 0, 0, 0};
  ctx->log_sites.clear();
  return FEATFIX_OK;
}

featfix_status featfix_set_forward_mask(featfix_ctx* ctx, int axis, const unsigned char* mask, int n) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  if (axis == FEATFIX_MASK_NONE) {
    if (ctx->fmask_axis != FEATFIX_MASK_NONE) graph_reset(ctx);
    ctx->fmask_axis = FEATFIX_MASK_NONE;
    return FEATFIX_OK;
  }
  if (axis != FEATFIX_MASK_TOKENS && axis != FEATFIX_MASK_CHANNELS) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "unknown mask axis");
  if (!mask) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "null mask");
  const int want = axis == FEATFIX_MASK_TOKENS ? ctx->Nt + ctx->Ni : ctx->C;
  if (n != want) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "mask length " + std::to_string(n) + ", expected " + std::to_string(want));
  FF_CK(cudaStreamSynchronize(ctx->user_st));
  graph_reset(ctx);
  std::vector<unsigned char> h;
  unsigned char** dst;
  if (axis == FEATFIX_MASK_TOKENS) {  // per token row of every model sample
    h.assign((size_t)ctx->T, 0);
    for (int b = 0; b < ctx->Bm; ++b)
      for (int t = 0; t < n; ++t) h[(size_t)featfix_token_row(&ctx->d, b, t)] = mask[t] ? 1 : 0;
    dst = &ctx->d_rmask;
  } else {
    h.assign(mask, mask + n);
    for (auto& v : h) v = v ? 1 : 0;
    dst = &ctx->d_cmask;
  }
  if (!*dst) FF_TRY(alloc(ctx, (void**)dst, h.size()));
  FF_CK(cudaMemcpy(*dst, h.data(), h.size(), cudaMemcpyHostToDevice));
  ctx->fmask_axis = axis;
  return FEATFIX_OK;
}

featfix_status featfix_get_plan(featfix_ctx* ctx, unsigned char* kinds, int* k_eff, double* weights) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  if (!ctx->sched) return fail(ctx, FEATFIX_ERR_STATE, "no schedule");
  if (kinds) std::memcpy(kinds, ctx->kinds.data(), ctx->kinds.size());
  if (k_eff) std::memcpy(k_eff, ctx->keff.data(), ctx->keff.size() * sizeof(int));
  if (weights) std::memcpy(weights, ctx->wts.data(), ctx->wts.size() * sizeof(double));
  return FEATFIX_OK;
}

featfix_status featfix_step(featfix_ctx* ctx, float* latent, int i, const void* cond) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  if (!latent || !cond) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "null latent or cond");
  if (!ctx->sched) return fail(ctx, FEATFIX_ERR_STATE, "featfix_set_schedule first");
  if (i != 0 && i != ctx->next_step) return fail(ctx, FEATFIX_ERR_STATE, "step out of order");
  if (i >= ctx->steps) return fail(ctx, FEATFIX_ERR_STATE, "step beyond the schedule");
  FF_TRY(compute_mods(ctx, cond, i, i + 1));
  return step_body(ctx, latent, i, cond);
}

featfix_status featfix_sample(featfix_ctx* ctx, unsigned long long seed, int steps, const void* cond,
                              float* latent_out) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  if (!ctx->sched) return fail(ctx, FEATFIX_ERR_STATE, "featfix_set_schedule first");
  if (steps != ctx->steps) return fail(ctx, FEATFIX_ERR_SCHEDULE, "steps differ from the schedule");
  if (!latent_out || !cond) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "null latent or cond");
  FF_CK(cudaMemcpyAsync(ctx->g_cond, cond, ctx->cond_bytes, cudaMemcpyDeviceToDevice, ctx->user_st));
  {
    KTimer tm(ctx, FEATFIX_KCLASS_OTHER, 0);
    FF_CK(launch_noise(seed, ctx->g_lat, ctx->lat_elems, ctx->user_st));
  }
  if (!ctx->graph_ok) FF_TRY(build_graph(ctx));
  FF_CK(cudaGraphLaunch(ctx->gexec, ctx->user_st));
  count_launches(ctx->graph_kernels);
  FF_CK(cudaMemcpyAsync(latent_out, ctx->g_lat, (size_t)ctx->lat_elems * 4, cudaMemcpyDeviceToDevice, ctx->user_st));
  bool timed = false;
  for (int k = 0; k < NKCLASS; ++k) timed |= ctx->timing[k];
  if (timed) {
    FF_CK(cudaStreamSynchronize(ctx->user_st));
    timing_take_graph(ctx);
  }
  return FEATFIX_OK;
}

featfix_status featfix_sample_host(featfix_ctx* ctx, unsigned long long seed, int steps, const void* cond_host,
                                   float* latent_out_host) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  if (!cond_host || !latent_out_host) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "null host buffer");
  if (!ctx->h_latent) FF_TRY(alloc(ctx, (void**)&ctx->h_latent, (size_t)ctx->lat_elems * sizeof(float)));
  if (!ctx->h_cond) FF_TRY(alloc(ctx, &ctx->h_cond, ctx->cond_bytes));
  FF_CK(cudaMemcpyAsync(ctx->h_cond, cond_host, ctx->cond_bytes, cudaMemcpyHostToDevice, ctx->user_st));
  FF_TRY(featfix_sample(ctx, seed, steps, ctx->h_cond, ctx->h_latent));
  FF_CK(cudaMemcpyAsync(latent_out_host, ctx->h_latent, (size_t)ctx->lat_elems * sizeof(float),
                        cudaMemcpyDeviceToHost, ctx->user_st));
  FF_CK(cudaStreamSynchronize(ctx->user_st));
  return FEATFIX_OK;
}

featfix_status featfix_get_log(featfix_ctx* ctx, featfix_site_log* out, int cap, int* n, featfix_counters* counters) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  FF_CK(cudaStreamSynchronize(ctx->user_st));
  const unsigned int wd = gemm_tc_watchdog_take() | (attention_tc_watchdog_take() << 8);
  if (wd) return fail(ctx, FEATFIX_ERR_CUDA, "tensor-core kernel watchdog fired (code " + std::to_string(wd) + ")");
  const int avail = (int)ctx->log_sites.size();
  if (n) *n = avail;
  if (counters) *counters = ctx->cnt;
  const int k = std::min(std::max(cap, 0), avail);
  if (k > 0 && out) {
    std::vector<double> sums((size_t)k * 4);
    FF_CK(cudaMemcpy(sums.data(), ctx->dsums, sums.size() * sizeof(double), cudaMemcpyDeviceToHost));
    for (int j = 0; j < k; ++j) {
      const double* q = &sums[(size_t)j * 4];
      out[j].step = ctx->log_sites[j].first;
      out[j].layer = ctx->log_sites[j].second;
      out[j].rel_l1 = q[0] / (q[1] + 1e-8);
      out[j].rel_l2 = std::sqrt(q[2]) / (std::sqrt(q[3]) + 1e-8);
      out[j].norm_l1_f = q[1];
      out[j].norm_l2_f = std::sqrt(q[3]);
    }
  }
  return FEATFIX_OK;
}

featfix_status featfix_debug_capture(featfix_ctx* ctx, int step, int layer, void* dev_in, void* dev_out) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  if (step < 0) {
    ctx->caps.clear();
    graph_reset(ctx);
    return FEATFIX_OK;
  }
  if (layer < 0 || layer >= ctx->L || (!dev_in && !dev_out)) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "bad capture");
  if (ctx->caps.size() >= 64) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "too many captures");
  ctx->caps.push_back({step, layer, dev_in, dev_out, {nullptr, nullptr, nullptr, nullptr}, 0});
  graph_reset(ctx);
  return FEATFIX_OK;
}

featfix_status featfix_debug_watchdog_probe(featfix_ctx* ctx, unsigned long long limit_ns) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  if (limit_ns < 1000ull || limit_ns > 1000000000ull) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "probe limit out of range");
  FF_CK(watchdog_probe(limit_ns, ctx->user_st));
  return FEATFIX_OK;
}

featfix_status featfix_debug_capture_history(featfix_ctx* ctx, int step, int layer, void* const* dev_slots, int n) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  if (step < 0 || layer < 0 || layer >= ctx->L || n < 1 || n > 4 || !dev_slots)
    return fail(ctx, FEATFIX_ERR_INVALID_ARG, "bad history capture");
  for (int j = 0; j < n; ++j)
    if (!dev_slots[j]) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "bad history capture");
  if (ctx->caps.size() >= 64) return fail(ctx, FEATFIX_ERR_INVALID_ARG, "too many captures");
  Capture cp = {step, layer, nullptr, nullptr, {nullptr, nullptr, nullptr, nullptr}, n};
  for (int j = 0; j < n; ++j) cp.hist[j] = dev_slots[j];
  ctx->caps.push_back(cp);
  graph_reset(ctx);
  return FEATFIX_OK;
}

featfix_status featfix_debug_block(featfix_ctx* ctx, int step, int layer, const void* dev_in, void* dev_out,
                                   const void* cond) {
  if (!ctx) return FEATFIX_ERR_INVALID_ARG;
  if (!ctx->sched) return fail(ctx, FEATFIX_ERR_STATE, "featfix_set_schedule first");
  if (step < 0 || step >= ctx->steps || layer < 0 || layer >= ctx->L || !dev_in || !dev_out || !cond)
    return fail(ctx, FEATFIX_ERR_INVALID_ARG, "bad debug block request");
  // modulations of `step` into the spare row block of the table
  const int spare = std::max(ctx->n_need, 1);
  const int saved = ctx->need_row[step];
  ctx->need_row[step] = spare;
  featfix_status s = compute_mods(ctx, cond, step, step + 1);
  ctx->need_row[step] = saved;
  if (s != FEATFIX_OK) return s;
  ctx->mod_row_override = spare;
  ctx->ln_src[0] = ctx->ln_src[1] = false;
  ctx->ln_next = false;
  s = exact_block(ctx, step, layer, dev_in, dev_out, nullptr);
  ctx->mod_row_override = -1;
  return s;
}

featfix_status featfix_kernel_timing(featfix_ctx* ctx, int kclass, int on) {
  if (!ctx || kclass < 0 || kclass >= NKCLASS) return FEATFIX_ERR_INVALID_ARG;
  FF_CK(cudaStreamSynchronize(ctx->user_st));
  timing_drain(ctx);
  if (ctx->timing[kclass] != (on != 0)) graph_reset(ctx);
  ctx->timing[kclass] = on != 0;
  ctx->tms[kclass] = 0;
  ctx->twork[kclass] = 0;
  ctx->tcount[kclass] = 0;
  return FEATFIX_OK;
}

featfix_status featfix_kernel_time(featfix_ctx* ctx, int kclass, double* ms, long long* launches, double* work) {
  if (!ctx || kclass < 0 || kclass >= NKCLASS) return FEATFIX_ERR_INVALID_ARG;
  FF_CK(cudaStreamSynchronize(ctx->user_st));
  timing_drain(ctx);
  if (ms) *ms = ctx->tms[kclass];
  if (launches) *launches = ctx->tcount[kclass];
  if (work) *work = ctx->twork[kclass];
  return FEATFIX_OK;
}

}  // extern "C"
