// Internal declarations shared by the FeatFix CUDA translation units.
// Not part of the public ABI (include/featfix.h, include/featfix_ops.h).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace ff {

enum DType : int { F32 = 0, BF16 = 1 };
typedef __nv_bfloat16 bf16;

static inline int dsize(DType t) { return t == F32 ? 4 : 2; }

// ---------------------------------------------------------------------------
// element conversion and 16-byte vectors
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }
template <class T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float x) { return __float2bfloat16_rn(x); }

template <class T> struct VecN { static constexpr int n = 16 / (int)sizeof(T); };

__device__ __forceinline__ void ld16(const float* p, float (&v)[4]) {
  float4 q = *reinterpret_cast<const float4*>(p);
  v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
}
__device__ __forceinline__ void ld16(const bf16* p, float (&v)[8]) {
  uint4 q = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&q);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 f = __bfloat1622float2(h[i]);
    v[2 * i] = f.x;
    v[2 * i + 1] = f.y;
  }
}
// a 16-byte vector already in registers, as floats
__device__ __forceinline__ void unpack16(const uint4& q, float (&v)[4]) {
  v[0] = __uint_as_float(q.x); v[1] = __uint_as_float(q.y); v[2] = __uint_as_float(q.z); v[3] = __uint_as_float(q.w);
}
__device__ __forceinline__ void unpack16(const uint4& q, float (&v)[8]) {
  const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[i]));
    v[2 * i] = f.x;
    v[2 * i + 1] = f.y;
  }
}
__device__ __forceinline__ void st16(float* p, const float (&v)[4]) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
}
__device__ __forceinline__ void st16(bf16* p, const float (&v)[8]) {
  uint4 q;
  __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&q);
#pragma unroll
  for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
  *reinterpret_cast<uint4*>(p) = q;
}
// round-trip through the storage type (value as it is stored)
__device__ __forceinline__ float round_to(float x, float*) { return x; }
__device__ __forceinline__ float round_to(float x, bf16*) { return __bfloat162float(__float2bfloat16_rn(x)); }

__device__ __forceinline__ float gelu_tanh(float x) {
  const float k0 = 0.7978845608028654f;  // sqrt(2/pi)
  return 0.5f * x * (1.0f + tanhf(k0 * (x + 0.044715f * x * x * x)));
}
// Same GELU through the hardware tanh approximation (tanh.approx.f32, about
// 2^-11 relative error): for bf16 outputs, whose rounding is 2^-9.
__device__ __forceinline__ float gelu_tanh_fast(float x) {
  const float k0 = 0.7978845608028654f;
  float t;
  asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(k0 * (x + 0.044715f * x * x * x)));
  return 0.5f * x * (1.0f + t);
}
__device__ __forceinline__ float silu(float x) { return x / (1.0f + expf(-x)); }

// ---------------------------------------------------------------------------
// fused GEMM epilogue: y = act(acc + bias); rope; out = resid + gate * y;
// hist_out = stored(out) - hist_base
// ---------------------------------------------------------------------------
struct EpiArgs {
  const void* bias;      // [N] model dtype (nullable)
  int act;               // 0 identity, 1 GELU(tanh), 2 SiLU
  int act_col0;          // activation only on columns >= act_col0
  const float* gate;     // gate rows (nullable): gate[b * gate_stride + n]
  int gate_stride;
  int seg_split;         // batch of row r: r < seg_split ? r / rpb0 : (r - seg_split) / rpb1
  int rpb0, rpb1;
  const void* resid;     // [M, ld_resid] model dtype (nullable); out = resid + (gate ? gate*y : y)
  int ld_resid;
  void* out;             // [M, ldo]
  int ldo;
  int out_f32;           // out (and out2) are float32 instead of the model dtype
  int split_col;         // columns >= split_col go to out2 at column n - split_col (N if unused)
  void* out2;
  int ldo2;
  const void* hist_base; // [M, ldo] model dtype (nullable)
  void* hist_out;        // [M, ldo] model dtype: stored(out) - hist_base
  const float2* rope;    // (cos, sin) table [rope_period][rope_half] (nullable)
  int rope_row0;         // rows >= rope_row0 are rotated
  int rope_period;       // image tokens per sample
  int rope_cols;         // columns < rope_cols (q and k) are rotated
  int rope_hd;           // head width d (pairs (2j, 2j+1) within a head)
  // adaLN LayerNorm of the next layer fused across two GEMMs (bf16 tensor-
  // core path; rows map to samples as for the gate).  With
  //   LN(x) (1 + s) + sh = rstd (x - mean) (1 + s) + sh
  // the next layer's product with W splits into
  //   rstd * [x (1 + s)] W^T - rstd * mean * [(1 + s) W^T] + sh W^T.
  // Producer (ln_out non-null): the stored output row also goes out scaled,
  // ln_out = stored(out) * (1 + ln_scale[b, n]) (row stride ldo), and every
  // 32-column chunk of the stored row leaves (sum, sum of squared deviations
  // from the chunk mean) in ln_stats[m * ln_slots + n / 32].
  const float* ln_scale;
  int ln_stride;
  void* ln_out;
  float2* ln_stats;
  int ln_slots;
  // Consumer (ln_in non-null): the A operand is such a scaled copy, and
  //   acc <- rstd * acc - rstd * mean * ln_c[b, n] + ln_d[b, n]
  // comes before the bias; mean and rstd (eps 1e-6) of row m combine its
  // ln_slots chunk statistics over ln_cols columns; ln_c = (1 + s) W^T and
  // ln_d = sh W^T per sample, rows of ln_cd_stride floats.
  const float2* ln_in;
  int ln_cols;
  const float* ln_c;
  const float* ln_d;
  int ln_cd_stride;
};

static inline EpiArgs epi_plain(void* out, int ldo) {
  EpiArgs e = {};
  e.out = out;
  e.ldo = ldo;
  e.act_col0 = 0;
  e.split_col = 0x7fffffff;
  e.rpb0 = 1;
  e.rpb1 = 1;
  return e;
}

__device__ __forceinline__ int epi_batch(const EpiArgs& e, int r) {
  return r < e.seg_split ? r / e.rpb0 : (r - e.seg_split) / e.rpb1;
}

// RoPE on q / k columns of image rows, then the activation.
template <class T, int CH>
__device__ __forceinline__ void epi_rope_act(const EpiArgs& e, int m, int n0, float (&v)[CH]) {
  if (e.rope && m >= e.rope_row0 && n0 < e.rope_cols) {
    const int tok = (m - e.rope_row0) % e.rope_period;
    const int half = e.rope_hd >> 1;
#pragma unroll
    for (int j = 0; j < CH; j += 2) {
      const int pair = ((n0 + j) % e.rope_hd) >> 1;
      const float2 cs = e.rope[(size_t)tok * half + pair];
      const float a = v[j], b = v[j + 1];
      v[j] = a * cs.x - b * cs.y;
      v[j + 1] = a * cs.y + b * cs.x;
    }
  }
  if (e.act == 1 && n0 >= e.act_col0) {
#pragma unroll
    for (int j = 0; j < CH; ++j) v[j] = sizeof(T) == 2 ? gelu_tanh_fast(v[j]) : gelu_tanh(v[j]);
  } else if (e.act == 2 && n0 >= e.act_col0) {
#pragma unroll
    for (int j = 0; j < CH; ++j) v[j] = silu(v[j]);
  }
}

// Applies the epilogue to CH consecutive accumulator columns n0 .. n0+CH-1
// of row m.  The chunk must not straddle split_col, act_col0 or rope_cols,
// and CH must be a multiple of the 16-byte vector width of T.  Columns >= N
// are skipped (N % vector width == 0).
// The part of the epilogue before the residual: y = gate * act(acc + bias),
// with RoPE applied to q / k columns.
// (rstd, rstd * mean) of row m for the fused LayerNorm's consumer, from the
// row's 32-column chunk statistics: mean = sum / C and
//   M2 = sum_i M2_i + sum_i 32 mean_i^2 - C mean^2.
__device__ __forceinline__ float2 ln_row(const EpiArgs& e, int m) {
  const float4* p = reinterpret_cast<const float4*>(e.ln_in + (size_t)m * e.ln_slots);
  float s1 = 0.f, s2 = 0.f, s3 = 0.f;
  for (int k = 0; k < e.ln_slots / 2; ++k) {
    const float4 q = __ldg(p + k);
    s1 += q.x + q.z;
    s2 += q.y + q.w;
    s3 = fmaf(q.x, q.x, fmaf(q.z, q.z, s3));
  }
  if (e.ln_slots & 1) {
    const float2 q = __ldg(e.ln_in + (size_t)m * e.ln_slots + e.ln_slots - 1);
    s1 += q.x;
    s2 += q.y;
    s3 = fmaf(q.x, q.x, s3);
  }
  const float C = (float)e.ln_cols;
  const float mean = s1 / C;
  const float m2 = fmaxf(s2 + s3 * (1.0f / 32.0f) - C * mean * mean, 0.f);
  const float rstd = rsqrtf(m2 / C + 1e-6f);
  return make_float2(rstd, rstd * mean);
}

// Consumer correction of CH accumulator columns n0.. of row m (sample b):
// v <- rstd * v - rstd * mean * ln_c + ln_d.
template <int CH>
__device__ __forceinline__ void ln_correct(const EpiArgs& e, int b, int n0, int N, float2 lnr, float (&v)[CH]) {
  const float* cr = e.ln_c + (size_t)b * e.ln_cd_stride + n0;
  const float* dr = e.ln_d + (size_t)b * e.ln_cd_stride + n0;
#pragma unroll
  for (int j = 0; j < CH; j += 4) {
    if (n0 + j < N) {
      const float4 c4 = __ldg(reinterpret_cast<const float4*>(cr + j));
      const float4 d4 = __ldg(reinterpret_cast<const float4*>(dr + j));
      v[j] = fmaf(lnr.x, v[j], fmaf(-lnr.y, c4.x, d4.x));
      v[j + 1] = fmaf(lnr.x, v[j + 1], fmaf(-lnr.y, c4.y, d4.y));
      v[j + 2] = fmaf(lnr.x, v[j + 2], fmaf(-lnr.y, c4.z, d4.z));
      v[j + 3] = fmaf(lnr.x, v[j + 3], fmaf(-lnr.y, c4.w, d4.w));
    }
  }
}

// Producer side for CH stored values x of row m (sample b), columns n0..:
// writes ln_out = x * (1 + ln_scale) and returns the chunk's (sum, sum of
// squared deviations from its mean).
template <int CH>
__device__ __forceinline__ float2 ln_emit(const EpiArgs& e, int m, int b, int n0, const float (&x)[CH]) {
  const float* sc = e.ln_scale + (size_t)b * e.ln_stride + n0;
  bf16* o = reinterpret_cast<bf16*>(e.ln_out) + (size_t)m * e.ldo + n0;
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < CH; j += 8) {
    const float4 a4 = __ldg(reinterpret_cast<const float4*>(sc + j));
    const float4 b4 = __ldg(reinterpret_cast<const float4*>(sc + j + 4));
    const float t[8] = {x[j] * (1.f + a4.x), x[j + 1] * (1.f + a4.y), x[j + 2] * (1.f + a4.z),
                        x[j + 3] * (1.f + a4.w), x[j + 4] * (1.f + b4.x), x[j + 5] * (1.f + b4.y),
                        x[j + 6] * (1.f + b4.z), x[j + 7] * (1.f + b4.w)};
    st16(o + j, t);
#pragma unroll
    for (int q = 0; q < 8; ++q) s += x[j + q];
  }
  const float mean = s * (1.0f / CH);
  float m2 = 0.f;
#pragma unroll
  for (int j = 0; j < CH; ++j) {
    const float d = x[j] - mean;
    m2 = fmaf(d, d, m2);
  }
  return make_float2(s, m2);
}

// Two 16-column halves of a 32-column chunk held by lanes l and l ^ 1
// (every lane of the warp calls this): the chunk's (sum, M2) on both lanes.
__device__ __forceinline__ float2 ln_pair(float2 st) {
  const float os = __shfl_xor_sync(0xffffffffu, st.x, 1);
  const float om = __shfl_xor_sync(0xffffffffu, st.y, 1);
  const float d = (st.x - os) * (1.0f / 16.0f);
  return make_float2(st.x + os, st.y + om + d * d * 8.0f);
}

__device__ __forceinline__ void ln_put(const EpiArgs& e, int m, int n0, float2 st) {
  e.ln_stats[(size_t)m * e.ln_slots + (n0 >> 5)] = st;
}

// LNM (compile time): which sides of the fused LayerNorm the caller's
// kernel instance handles -- bit 0 consumer (ln_in), bit 1 producer (ln_out).
template <class T, int CH, int LNM = 3>
__device__ __forceinline__ void epi_math(const EpiArgs& e, int m, int n0, int N, float (&v)[CH],
                                         float2 lnr = make_float2(1.f, 0.f)) {
  constexpr int V = VecN<T>::n;
  if ((LNM & 1) && e.ln_in) ln_correct<CH>(e, epi_batch(e, m), n0, N, lnr, v);
  if (e.bias) {
    const T* b = reinterpret_cast<const T*>(e.bias);
#pragma unroll
    for (int j = 0; j < CH; j += V) {
      if (n0 + j < N) {
        float bb[V];
        ld16(b + n0 + j, bb);
#pragma unroll
        for (int q = 0; q < V; ++q) v[j + q] += bb[q];
      }
    }
  }
  epi_rope_act<T, CH>(e, m, n0, v);
  if (e.gate) {
    const float* g = e.gate + (size_t)epi_batch(e, m) * e.gate_stride + n0;
#pragma unroll
    for (int j = 0; j < CH; j += 4) {
      if (n0 + j < N) {
        float4 gg = *reinterpret_cast<const float4*>(g + j);
        v[j] *= gg.x; v[j + 1] *= gg.y; v[j + 2] *= gg.z; v[j + 3] *= gg.w;
      }
    }
  }
}

// Returns the chunk's (sum, M2) of the stored values when the output feeds a
// fused LayerNorm (ln_out; bf16, chunks of 16 or 32 whole columns), else 0.
template <class T, int CH, int LNM = 3>
__device__ __forceinline__ float2 epi_chunk(const EpiArgs& e, int m, int n0, int N, float (&v)[CH],
                                            float2 lnr = make_float2(1.f, 0.f)) {
  constexpr int V = VecN<T>::n;
  epi_math<T, CH, LNM>(e, m, n0, N, v, lnr);
  if (e.resid) {
    const T* rs = reinterpret_cast<const T*>(e.resid) + (size_t)m * e.ld_resid + n0;
#pragma unroll
    for (int j = 0; j < CH; j += V) {
      if (n0 + j < N) {
        float rr[V];
        ld16(rs + j, rr);
#pragma unroll
        for (int q = 0; q < V; ++q) v[j + q] += rr[q];
      }
    }
  }
  const bool second = n0 >= e.split_col;
  const int col = second ? n0 - e.split_col : n0;
  const int ld = second ? e.ldo2 : e.ldo;
  void* obase = second ? e.out2 : e.out;
  if (e.out_f32) {
    float* o = reinterpret_cast<float*>(obase) + (size_t)m * ld + col;
#pragma unroll
    for (int j = 0; j < CH; j += 4) {
      if (n0 + j < N) {
        float t[4] = {v[j], v[j + 1], v[j + 2], v[j + 3]};
        st16(o + j, t);
      }
    }
  } else {
    T* o = reinterpret_cast<T*>(obase) + (size_t)m * ld + col;
#pragma unroll
    for (int j = 0; j < CH; j += V) {
      if (n0 + j < N) {
        float t[V];
#pragma unroll
        for (int q = 0; q < V; ++q) t[q] = v[j + q];
        st16(o + j, t);
      }
    }
  }
  if (e.hist_out) {
    const T* hb = reinterpret_cast<const T*>(e.hist_base) + (size_t)m * e.ldo + n0;
    T* ho = reinterpret_cast<T*>(e.hist_out) + (size_t)m * e.ldo + n0;
#pragma unroll
    for (int j = 0; j < CH; j += V) {
      if (n0 + j < N) {
        float u[V], t[V];
        ld16(hb + j, u);
#pragma unroll
        for (int q = 0; q < V; ++q) t[q] = round_to(v[j + q], (T*)nullptr) - u[q];
        st16(ho + j, t);
      }
    }
  }
  if constexpr (sizeof(T) == 2 && CH % 8 == 0 && (LNM & 2) != 0) {
    if (e.ln_out && !e.out_f32 && n0 + CH <= N) {
      float x[CH];
#pragma unroll
      for (int j = 0; j < CH; ++j) x[j] = round_to(v[j], (T*)nullptr);
      return ln_emit<CH>(e, m, epi_batch(e, m), n0, x);
    }
  }
  return make_float2(0.f, 0.f);
}

// ---------------------------------------------------------------------------
// programmatic dependent launch: a kernel launched with launch_pdl may start
// while the previous kernel on the stream is still finishing.  It lets its
// own dependents launch (pdl_trigger) and then waits for the previous
// kernel to complete, memory included (pdl_wait), before it touches global
// memory.  Both are no-ops in a kernel launched the ordinary way.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
static inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                                     Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ---------------------------------------------------------------------------
// launchers (return the launch error; work is asynchronous on `s`)
// ---------------------------------------------------------------------------
struct Hist4 { const void* p[4]; };
// The history entries of a run of consecutive drafted blocks (at most
// SEG_MAX blocks, K_eff + 1 entries each, newest first).
constexpr int SEG_MAX = 64;
struct HistSeg { const void* p[SEG_MAX][4]; };

// Process-wide count of kernels this library has launched.
void count_launches(long long n);
long long launches_total();
inline cudaError_t launched() {
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_draft(DType dt, void* x, const Hist4& h, const float* w, int nt, long long n, cudaStream_t s);
// x <- x + sum_{b < nblk} sum_j w_j h.p[b][j]: the per-block drafts of nblk
// consecutive blocks (Eq. 2 with the same weights for every block) chained
// in one pass, in fp32, rounded once.
cudaError_t launch_draft_seg(DType dt, void* x, const HistSeg& h, int nblk, const float* w, int nt, long long n,
                             cudaStream_t s);
cudaError_t launch_diff(DType dt, const void* a, const void* b, void* out, long long n, cudaStream_t s);
size_t verify_workspace_bytes(long long n);
// Queries how many paid-check clusters are resident at once (the launched
// grid); done on first use, or here ahead of any stream capture.
void verify_prepare();
// Partial forwarding at a site: out <- h_f on selected rows (rmask, per
// token row) or columns (cmask), h_d elsewhere; row width C.
struct FwdMix {
  void* out;
  const unsigned char* rmask;
  const unsigned char* cmask;
  int C;
};
// done_ctr: a zeroed counter owned by the caller turns the reduction into
// one launch (the last cluster sums the partials and resets the counter);
// without it a second one-block launch sums them.
cudaError_t launch_verify(DType dt, void* u, const Hist4& h, const float* w, int nt, const void* hf, long long n,
                          int write_draft, double* sums, void* ws, cudaStream_t s,
                          const FwdMix* mix = nullptr, unsigned int* done_ctr = nullptr);
// Operand rows of the fused-LayerNorm correction GEMMs (see k_ln_ab).
cudaError_t launch_ln_ab(DType dt, const float* mod, long long mod_stride, int rows, int C, const int2* jobs,
                         int njobs, void* out, long long job_stride, cudaStream_t s);
cudaError_t launch_ln_mod(DType dt, const void* x, void* out, long long rows, int C, const float* shift,
                          const float* scale, int mod_stride, int seg_split, int rpb0, int rpb1, cudaStream_t s);
// Sinusoidal features of S model times (device array) -> [S, 256] in dt.
cudaError_t launch_sinusoid_table(DType dt, const float* times, int S, void* out, cudaStream_t s);
// SiLU(temb[s] + y_emb[label_b]) for every (step s, sample b): rows s*B + b of
// `all` ([S*B, C], dt); rows of steps with need_row[s] >= 0 also go to
// need[(need_row[s]*B + b)] (gathered table).
cudaError_t launch_cond_table(DType dt, const float* temb, const void* y_emb, const int* labels, int S, int B, int C,
                              const int* need_row, void* all, void* need, cudaStream_t s);
cudaError_t launch_cond_finish(DType wt, const float* e, const void* y_emb, const int* labels, int B, int C,
                               float* c_out, float* csilu_out, cudaStream_t s);
cudaError_t launch_patchify(DType dt, const float* latent, int B_lat, int B_model, int Cin, int F, int H, int W,
                            int p, int pt, void* out, cudaStream_t s);
cudaError_t launch_convert(DType dt, const float* in, void* out, long long n, cudaStream_t s);
cudaError_t launch_sampler(const float* model_out, float* latent, int B_lat, int cfg, float cfg_scale, int Cin,
                           int Cout, int F, int H, int W, int p, int pt, float c1, float c2, cudaStream_t s);
cudaError_t launch_noise(unsigned long long seed, float* out, long long n, cudaStream_t s);
cudaError_t launch_pos2d(DType dt, void* out, int B, int gh, int gw, int C, cudaStream_t s);

// dense layers: out = epilogue(A[M,K] W[N,K]^T)
cudaError_t gemm_simt(DType dt, int M, int N, int K, const void* A, int lda, const void* W, int ldw,
                      const EpiArgs& e, cudaStream_t s);
cudaError_t gemm_tc(int M, int N, int K, const void* A, int lda, const void* W, int ldw, const EpiArgs& e,
                    cudaStream_t s);
// Two problems of the same N and K (A0 W0^T with epilogue e0 over M0 rows and
// A1 W1^T with e1 over M1 rows, the same lda / ldw) in one persistent launch
// where possible: the second stream's few tiles fill the wave of the first.
cudaError_t gemm_tc_grouped(int M0, const void* A0, const void* W0, const EpiArgs& e0, int M1, const void* A1,
                            const void* W1, const EpiArgs& e1, int N, int K, int lda, int ldw, cudaStream_t s);
unsigned int gemm_tc_watchdog_take();
cudaError_t watchdog_probe(unsigned long long limit_ns, cudaStream_t s);

// attention over the token-row layout (see featfix_token_row)
struct AttnArgs {
  const void* q; const void* k; const void* v;  // base pointers (column offsets applied)
  int ld_qkv;
  void* out; int ld_out;
  int B, Nt, Ni, H, hd;
};
cudaError_t attention(DType dt, const AttnArgs& a, cudaStream_t s);
cudaError_t attention_tc(const AttnArgs& a, cudaStream_t s);
unsigned int attention_tc_watchdog_take();
cudaError_t attention_simt(DType dt, const AttnArgs& a, cudaStream_t s);

}  // namespace ff
