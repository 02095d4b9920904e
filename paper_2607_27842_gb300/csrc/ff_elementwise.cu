// Bandwidth-bound kernels of the FeatFix denoising step: the draft (Eq. 2),
// the fused paid check / forward (Eqs. 3-5), adaLN LayerNorm-modulation,
// conditioning tables, embedding, sampler update and the seeded latent.
#include "ff_common.cuh"

#include <cooperative_groups.h>
#include <math.h>

#include <atomic>

namespace cg = cooperative_groups;

namespace ff {

static std::atomic<long long> g_launches{0};
void count_launches(long long n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
long long launches_total() { return g_launches.load(std::memory_order_relaxed); }

static int g_num_sms = 0;
static int num_sms() {
  if (g_num_sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (g_num_sms <= 0) g_num_sms = 148;
  }
  return g_num_sms;
}

// ---------------------------------------------------------------------------
// Draft (Eq. 2, weight form): x <- x + sum_j w_j R_j.  One 16-byte vector per
// thread per iteration, every operand streamed once, grid-stride over a grid
// sized to a multiple of the SM count.
// ---------------------------------------------------------------------------
template <class T, int NT>
__device__ __forceinline__ void draft_vec(const T* __restrict__ xu, const Hist4& h, const float (&w)[4], long long i,
                                          float (&a)[VecN<T>::n]) {
  constexpr int V = VecN<T>::n;
  ld16(xu + i * V, a);
#pragma unroll
  for (int j = 0; j < NT; ++j) {
    float r[V];
    ld16(reinterpret_cast<const T*>(h.p[j]) + i * V, r);
#pragma unroll
    for (int q = 0; q < V; ++q) a[q] = __fmaf_rn(w[j], r[q], a[q]);
  }
}

template <class T, int NT>
__device__ __forceinline__ float draft_scalar(const T* xu, const Hist4& h, const float (&w)[4], long long i) {
  float a = to_f(xu[i]);
#pragma unroll
  for (int j = 0; j < NT; ++j) a = __fmaf_rn(w[j], to_f(reinterpret_cast<const T*>(h.p[j])[i]), a);
  return a;
}

template <class T, int NT>
__global__ void __launch_bounds__(256) k_draft(T* __restrict__ x, Hist4 h, float w0, float w1, float w2, float w3,
                                               long long n) {
  pdl_trigger();
  pdl_wait();
  constexpr int V = VecN<T>::n;
  const float w[4] = {w0, w1, w2, w3};
  const long long nvec = n / V;
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < nvec; i += stride) {
    float a[V];
    draft_vec<T, NT>(x, h, w, i, a);
    st16(x + i * V, a);
  }
  if (blockIdx.x == 0 && threadIdx.x < n - nvec * V) {
    const long long i = nvec * V + threadIdx.x;
    x[i] = from_f<T>(draft_scalar<T, NT>(x, h, w, i));
  }
}

static int stream_grid(long long nvec, int threads) {
  long long want = (nvec + threads - 1) / threads;
  long long cap = (long long)num_sms() * 8;
  if (want > cap) want = cap;
  if (want < 1) want = 1;
  return (int)want;
}

template <class T>
static cudaError_t draft_t(void* x, const Hist4& h, const float* w, int nt, long long n, cudaStream_t s) {
  const int grid = stream_grid(n / VecN<T>::n, 256);
  T* xp = reinterpret_cast<T*>(x);
  switch (nt) {
    case 1: launch_pdl(k_draft<T, 1>, grid, 256, 0, s, xp, h, w[0], w[1], w[2], w[3], n); break;
    case 2: launch_pdl(k_draft<T, 2>, grid, 256, 0, s, xp, h, w[0], w[1], w[2], w[3], n); break;
    case 3: launch_pdl(k_draft<T, 3>, grid, 256, 0, s, xp, h, w[0], w[1], w[2], w[3], n); break;
    case 4: launch_pdl(k_draft<T, 4>, grid, 256, 0, s, xp, h, w[0], w[1], w[2], w[3], n); break;
    default: return cudaErrorInvalidValue;
  }
  return launched();
}

cudaError_t launch_draft(DType dt, void* x, const Hist4& h, const float* w, int nt, long long n, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  return dt == F32 ? draft_t<float>(x, h, w, nt, n, s) : draft_t<bf16>(x, h, w, nt, n, s);
}

// A run of nblk drafted blocks in one pass: x <- x + sum_b sum_j w_j R_{b,j}.
// Each block's draft adds its forecast increment to the incoming state, so
// the run's blocks telescope; x is read and written once instead of once
// per block, and the sum stays in fp32 until the end.
template <class T, int NT>
__global__ void __launch_bounds__(256) k_draft_seg(T* __restrict__ x, const __grid_constant__ HistSeg h, int nblk,
                                                   float w0, float w1, float w2, float w3, long long n) {
  pdl_trigger();
  pdl_wait();
  constexpr int V = VecN<T>::n;
  const float w[4] = {w0, w1, w2, w3};
  const long long nvec = n / V;
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < nvec; i += stride) {
    float a[V];
    ld16(x + i * V, a);
    for (int b = 0; b < nblk; ++b) {
#pragma unroll
      for (int j = 0; j < NT; ++j) {
        float r[V];
        ld16(reinterpret_cast<const T*>(h.p[b][j]) + i * V, r);
#pragma unroll
        for (int q = 0; q < V; ++q) a[q] = __fmaf_rn(w[j], r[q], a[q]);
      }
    }
    st16(x + i * V, a);
  }
  if (blockIdx.x == 0 && threadIdx.x < n - nvec * V) {
    const long long i = nvec * V + threadIdx.x;
    float a = to_f(x[i]);
    for (int b = 0; b < nblk; ++b) {
#pragma unroll
      for (int j = 0; j < NT; ++j) a = __fmaf_rn(w[j], to_f(reinterpret_cast<const T*>(h.p[b][j])[i]), a);
    }
    x[i] = from_f<T>(a);
  }
}

template <class T>
static cudaError_t draft_seg_t(void* x, const HistSeg& h, int nblk, const float* w, int nt, long long n,
                               cudaStream_t s) {
  const int grid = stream_grid(n / VecN<T>::n, 256);
  T* xp = reinterpret_cast<T*>(x);
  switch (nt) {
    case 1: launch_pdl(k_draft_seg<T, 1>, grid, 256, 0, s, xp, h, nblk, w[0], w[1], w[2], w[3], n); break;
    case 2: launch_pdl(k_draft_seg<T, 2>, grid, 256, 0, s, xp, h, nblk, w[0], w[1], w[2], w[3], n); break;
    case 3: launch_pdl(k_draft_seg<T, 3>, grid, 256, 0, s, xp, h, nblk, w[0], w[1], w[2], w[3], n); break;
    case 4: launch_pdl(k_draft_seg<T, 4>, grid, 256, 0, s, xp, h, nblk, w[0], w[1], w[2], w[3], n); break;
    default: return cudaErrorInvalidValue;
  }
  return launched();
}

cudaError_t launch_draft_seg(DType dt, void* x, const HistSeg& h, int nblk, const float* w, int nt, long long n,
                             cudaStream_t s) {
  if (n <= 0 || nblk <= 0) return cudaSuccess;
  if (nblk > SEG_MAX) return cudaErrorInvalidValue;
  return dt == F32 ? draft_seg_t<float>(x, h, nblk, w, nt, n, s) : draft_seg_t<bf16>(x, h, nblk, w, nt, n, s);
}

// out = a - b elementwise (fp32 arithmetic, rounded to the storage type).
template <class T>
__global__ void __launch_bounds__(256) k_diff(const T* __restrict__ a, const T* __restrict__ b, T* __restrict__ out,
                                              long long n) {
  pdl_trigger();
  pdl_wait();
  constexpr int V = VecN<T>::n;
  const long long nvec = n / V;
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < nvec; i += stride) {
    float x[V], y[V];
    ld16(a + i * V, x);
    ld16(b + i * V, y);
#pragma unroll
    for (int q = 0; q < V; ++q) x[q] -= y[q];
    st16(out + i * V, x);
  }
  if (blockIdx.x == 0 && threadIdx.x < n - nvec * V) {
    const long long i = nvec * V + threadIdx.x;
    out[i] = from_f<T>(to_f(a[i]) - to_f(b[i]));
  }
}

cudaError_t launch_diff(DType dt, const void* a, const void* b, void* out, long long n, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  if (dt == F32) {
    launch_pdl(k_diff<float>, stream_grid(n / 4, 256), 256, 0, s, (const float*)a, (const float*)b, (float*)out, n);
  } else {
    launch_pdl(k_diff<bf16>, stream_grid(n / 8, 256), 256, 0, s, (const bf16*)a, (const bf16*)b, (bf16*)out, n);
  }
  return launched();
}

// ---------------------------------------------------------------------------
// Paid check + forward (Eqs. 3-5), fused so h_f is read once: each thread
// rebuilds h_d from u and the history exactly as k_draft does, accumulates
// |h_d - h_f|, |h_f|, (h_d - h_f)^2, h_f^2, and (Verify arm) stores h_d over
// u.  Reduction: warp shuffles, then shared memory, then the 8 CTAs of a
// thread-block cluster combine through distributed shared memory; one
// partial per cluster goes to the workspace and a one-block kernel adds the
// partials in a fixed order (deterministic run to run).
// ---------------------------------------------------------------------------
constexpr int VERIFY_THREADS = 256;
constexpr int VERIFY_CLUSTER = 8;

// Upper bound of the grid (and so of the partials in the workspace): up to
// four CTAs per SM, whole clusters.
static int verify_grid(long long n) {
  long long nvec = n / 4 + 1;
  long long want = (nvec + VERIFY_THREADS - 1) / VERIFY_THREADS;
  long long cap = (long long)num_sms() * 4;
  if (want > cap) want = cap;
  want = (want + VERIFY_CLUSTER - 1) / VERIFY_CLUSTER * VERIFY_CLUSTER;
  if (want < VERIFY_CLUSTER) want = VERIFY_CLUSTER;
  return (int)want;
}

size_t verify_workspace_bytes(long long n) {
  return (size_t)(verify_grid(n) / VERIFY_CLUSTER) * 4 * sizeof(double);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Partial forwarding (token- or channel-level arm): mix != nullptr gets
// h_f where the element's row (rmask) or column (cmask) is selected and h_d
// elsewhere; mix may be the h_f buffer itself (each element is read, then
// written, by the same thread).
template <class T, int NT>
__global__ void __cluster_dims__(VERIFY_CLUSTER, 1, 1) __launch_bounds__(VERIFY_THREADS, 4)
    k_verify(T* __restrict__ u, Hist4 h, float w0, float w1, float w2, float w3, const T* hf,
             long long n, int write_draft, double* __restrict__ partials, T* mix,
             const unsigned char* __restrict__ rmask, const unsigned char* __restrict__ cmask, int C,
             unsigned int* done_ctr, double* __restrict__ sums) {
  pdl_trigger();
  pdl_wait();
  constexpr int V = VecN<T>::n;
  const float w[4] = {w0, w1, w2, w3};
  float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
  const long long nvec = n / V;
  const long long stride = (long long)gridDim.x * blockDim.x;
  // One vector of u, the history and h_f, accumulated, stored (Verify) and
  // mixed (partial forwarding).
  auto one = [&](long long i, float (&a)[V], const float (&f)[V]) {
#pragma unroll
    for (int q = 0; q < V; ++q) {
      const float ad = round_to(a[q], (T*)nullptr);  // h_d as it would be forwarded
      const float d = ad - f[q];
      s0 += fabsf(d);
      s1 += fabsf(f[q]);
      s2 += d * d;
      s3 += f[q] * f[q];
    }
    if (write_draft) st16(u + i * V, a);
    if (mix) {  // C % V == 0: the vector lies in one row
      const long long e0 = i * V;
      const long long r = e0 / C;
      const int c0 = (int)(e0 - r * C);
      float o[V];
#pragma unroll
      for (int q = 0; q < V; ++q) o[q] = (rmask ? rmask[r] : cmask[c0 + q]) ? f[q] : a[q];
      st16(mix + i * V, o);
    }
  };
  // Two vectors per thread and iteration, all their loads issued before
  // either is used: the grid holds at most four CTAs per SM (the partials
  // stay small), so each thread keeps twice the bytes in flight instead.
  long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  for (; i + stride < nvec; i += 2 * stride) {
    float a[V], f[V], a2[V], f2[V];
    draft_vec<T, NT>(u, h, w, i, a);
    draft_vec<T, NT>(u, h, w, i + stride, a2);
    ld16(hf + i * V, f);
    ld16(hf + (i + stride) * V, f2);
    one(i, a, f);
    one(i + stride, a2, f2);
  }
  if (i < nvec) {
    float a[V], f[V];
    draft_vec<T, NT>(u, h, w, i, a);
    ld16(hf + i * V, f);
    one(i, a, f);
  }
  if (blockIdx.x == 0 && threadIdx.x < n - nvec * V) {
    const long long i = nvec * V + threadIdx.x;
    const float a = round_to(draft_scalar<T, NT>(u, h, w, i), (T*)nullptr);
    const float f = to_f(hf[i]);
    const float d = a - f;
    s0 += fabsf(d); s1 += fabsf(f); s2 += d * d; s3 += f * f;
    if (write_draft) u[i] = from_f<T>(a);
    if (mix) mix[i] = from_f<T>((rmask ? rmask[i / C] : cmask[i % C]) ? f : a);
  }
  s0 = warp_sum(s0); s1 = warp_sum(s1); s2 = warp_sum(s2); s3 = warp_sum(s3);
  __shared__ float wsum[VERIFY_THREADS / 32][4];
  __shared__ double bsum[4];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) { wsum[warp][0] = s0; wsum[warp][1] = s1; wsum[warp][2] = s2; wsum[warp][3] = s3; }
  __syncthreads();
  if (threadIdx.x < 4) {
    double t = 0.0;
    for (int k = 0; k < VERIFY_THREADS / 32; ++k) t += (double)wsum[k][threadIdx.x];
    bsum[threadIdx.x] = t;
  }
  cg::cluster_group cluster = cg::this_cluster();
  cluster.sync();
  if (cluster.block_rank() == 0 && threadIdx.x < 32) {
    if (threadIdx.x < 4) {
      double t = 0.0;
      for (unsigned r = 0; r < cluster.num_blocks(); ++r) {
        const double* rb = cluster.map_shared_rank(bsum, r);
        t += rb[threadIdx.x];
      }
      partials[(size_t)(blockIdx.x / VERIFY_CLUSTER) * 4 + threadIdx.x] = t;
      __threadfence();
    }
    // With a completion counter the last cluster to finish sums every
    // cluster's partials in index order (the same order whichever cluster
    // is last) and resets the counter for the next launch.
    if (done_ctr) {
      __syncwarp();
      const unsigned int nclusters = gridDim.x / VERIFY_CLUSTER;
      unsigned int last = 0;
      if (threadIdx.x == 0) last = atomicAdd(done_ctr, 1u) == nclusters - 1 ? 1u : 0u;
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence();
        if (threadIdx.x < 4) {
          const volatile double* vp = partials;
          double t = 0.0;
          for (unsigned k = 0; k < nclusters; ++k) t += vp[(size_t)k * 4 + threadIdx.x];
          sums[threadIdx.x] = t;
        }
        if (threadIdx.x == 0) *done_ctr = 0u;
      }
    }
  }
  cluster.sync();
}

__global__ void k_verify_finish(const double* __restrict__ partials, int nparts, double* __restrict__ sums) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x < 4) {
    double t = 0.0;
    for (int k = 0; k < nparts; ++k) t += partials[(size_t)k * 4 + threadIdx.x];
    sums[threadIdx.x] = t;
  }
}

// The launched grid: verify_grid's bound, cut to the clusters that are
// resident at once.  Clusters of 8 CTAs must fit in one GPC, so four CTAs
// per SM on every SM are not all co-resident; a grid sized to them left a
// second wave of a few clusters that ran alone (measured: the paid check at
// 0.6 of the copy rate, with drafts of the same size at 1.0).
template <class T, int NT>
static int verify_launch_grid(long long n) {
  static int resident = -1;  // clusters resident at once (per kernel instance)
  if (resident < 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(VERIFY_CLUSTER * 64);
    cfg.blockDim = dim3(VERIFY_THREADS);
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = VERIFY_CLUSTER;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int nc = 0;
    if (cudaOccupancyMaxActiveClusters(&nc, k_verify<T, NT>, &cfg) != cudaSuccess || nc <= 0) {
      cudaGetLastError();
      nc = 0;  // unknown: keep the bound
    }
    resident = nc;
  }
  int grid = verify_grid(n);
  if (resident > 0 && grid > resident * VERIFY_CLUSTER) grid = resident * VERIFY_CLUSTER;
  return grid;
}

void verify_prepare() {
  verify_launch_grid<float, 1>(1); verify_launch_grid<float, 2>(1);
  verify_launch_grid<float, 3>(1); verify_launch_grid<float, 4>(1);
  verify_launch_grid<bf16, 1>(1); verify_launch_grid<bf16, 2>(1);
  verify_launch_grid<bf16, 3>(1); verify_launch_grid<bf16, 4>(1);
}

template <class T>
static cudaError_t verify_t(void* u, const Hist4& h, const float* w, int nt, const void* hf, long long n,
                           int write_draft, double* sums, void* ws, cudaStream_t s, const FwdMix* fm,
                           unsigned int* done_ctr) {
  const int grid = nt == 1 ? verify_launch_grid<T, 1>(n) : nt == 2 ? verify_launch_grid<T, 2>(n)
                 : nt == 3 ? verify_launch_grid<T, 3>(n) : verify_launch_grid<T, 4>(n);
  double* parts = reinterpret_cast<double*>(ws);
  T* up = reinterpret_cast<T*>(u);
  const T* fp = reinterpret_cast<const T*>(hf);
  T* mx = fm ? reinterpret_cast<T*>(fm->out) : nullptr;
  const unsigned char* rm = fm ? fm->rmask : nullptr;
  const unsigned char* cm = fm ? fm->cmask : nullptr;
  const int C = fm ? fm->C : 1;
  if (mx && (C <= 0 || C % VecN<T>::n != 0 || (!rm && !cm) || n % C != 0)) return cudaErrorInvalidValue;
  switch (nt) {
    case 1: launch_pdl(k_verify<T, 1>, grid, VERIFY_THREADS, 0, s, up, h, w[0], w[1], w[2], w[3], fp, n, write_draft, parts, mx, rm, cm, C, done_ctr, sums); break;
    case 2: launch_pdl(k_verify<T, 2>, grid, VERIFY_THREADS, 0, s, up, h, w[0], w[1], w[2], w[3], fp, n, write_draft, parts, mx, rm, cm, C, done_ctr, sums); break;
    case 3: launch_pdl(k_verify<T, 3>, grid, VERIFY_THREADS, 0, s, up, h, w[0], w[1], w[2], w[3], fp, n, write_draft, parts, mx, rm, cm, C, done_ctr, sums); break;
    case 4: launch_pdl(k_verify<T, 4>, grid, VERIFY_THREADS, 0, s, up, h, w[0], w[1], w[2], w[3], fp, n, write_draft, parts, mx, rm, cm, C, done_ctr, sums); break;
    default: return cudaErrorInvalidValue;
  }
  cudaError_t e = launched();
  if (e != cudaSuccess || done_ctr) return e;
  launch_pdl(k_verify_finish, 1, 32, 0, s, parts, grid / VERIFY_CLUSTER, sums);
  return launched();
}

cudaError_t launch_verify(DType dt, void* u, const Hist4& h, const float* w, int nt, const void* hf, long long n,
                          int write_draft, double* sums, void* ws, cudaStream_t s, const FwdMix* mix,
                          unsigned int* done_ctr) {
  if (n <= 0) return cudaErrorInvalidValue;
  return dt == F32 ? verify_t<float>(u, h, w, nt, hf, n, write_draft, sums, ws, s, mix, done_ctr)
                   : verify_t<bf16>(u, h, w, nt, hf, n, write_draft, sums, ws, s, mix, done_ctr);
}

// ---------------------------------------------------------------------------
// Operand rows of the fused-LayerNorm correction GEMMs: for job j (one
// LayerNorm of one block and stream) and modulation row r,
//   out[j][2r] = 1 + scale_r,  out[j][2r + 1] = shift_r
// (columns jobs[j].x and jobs[j].y of the row), so one GEMM with the layer's
// weight gives (1 + s) W^T and sh W^T interleaved.
// ---------------------------------------------------------------------------
template <class T>
__global__ void __launch_bounds__(256) k_ln_ab(const float* __restrict__ mod, long long mod_stride, int C,
                                               const int2* __restrict__ jobs, T* __restrict__ out,
                                               long long job_stride) {
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x, j = blockIdx.y;
  const int2 jc = jobs[j];
  const float* sc = mod + (size_t)r * mod_stride + jc.x;
  const float* sh = mod + (size_t)r * mod_stride + jc.y;
  T* o = out + (size_t)j * job_stride + (size_t)2 * r * C;
  for (int c = threadIdx.x; c < C; c += blockDim.x) {
    o[c] = from_f<T>(1.0f + sc[c]);
    o[C + c] = from_f<T>(sh[c]);
  }
}

cudaError_t launch_ln_ab(DType dt, const float* mod, long long mod_stride, int rows, int C, const int2* jobs,
                         int njobs, void* out, long long job_stride, cudaStream_t s) {
  if (rows <= 0 || njobs <= 0) return cudaSuccess;
  const dim3 grid(rows, njobs);
  if (dt == F32)
    launch_pdl(k_ln_ab<float>, grid, dim3(256), 0, s, mod, mod_stride, C, jobs, (float*)out, job_stride);
  else
    launch_pdl(k_ln_ab<bf16>, grid, dim3(256), 0, s, mod, mod_stride, C, jobs, (bf16*)out, job_stride);
  return launched();
}

// ---------------------------------------------------------------------------
// adaLN branch input: LN(x) (no affine, eps 1e-6) * (1 + scale_b) + shift_b.
// One warp per row, the row held in registers (NCH 16-byte vectors per
// lane): one global read, exact two-pass mean / variance, one write.
// ---------------------------------------------------------------------------
// One warp per row (8 rows per block, for row counts that fill about two
// waves at most); the block first stages the shift /
// scale vectors of its first row's sample in shared memory (coalesced, read
// back by every warp of that sample instead of 4 x 16 B per lane per chunk
// from global memory).  Rows of up to six vectors per lane are held to 64
// registers, so four blocks share an SM (4096 rows of 1152: one wave).
template <class T, int NCH>
__global__ void __launch_bounds__(256, NCH <= 6 ? 4 : 1) k_ln_mod1(const T* __restrict__ x, T* __restrict__ out, long long rows, int C,
                                                const float* __restrict__ shift, const float* __restrict__ scale,
                                                int mod_stride, int seg_split, int rpb0, int rpb1) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float4 smod4[];                  // [2 * C / 4]: shift, then scale
  float* smod = reinterpret_cast<float*>(smod4);
  constexpr int V = VecN<T>::n;
  const long long r0 = (long long)blockIdx.x * 8;
  const int b0 = (int)(r0 < seg_split ? r0 / rpb0 : (r0 - seg_split) / rpb1);
  {
    const float4* sh4 = reinterpret_cast<const float4*>(shift + (size_t)b0 * mod_stride);
    const float4* sc4 = reinterpret_cast<const float4*>(scale + (size_t)b0 * mod_stride);
    for (int i = threadIdx.x; i < C / 4; i += blockDim.x) {
      smod4[i] = sh4[i];
      smod4[C / 4 + i] = sc4[i];
    }
  }
  __syncthreads();
  const long long r = r0 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const T* xr = x + r * C;
  const int nv = C / V;
  float a[NCH][V];
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < NCH; ++j) {
    const int k = lane + 32 * j;
    if (k < nv) {
      ld16(xr + k * V, a[j]);
#pragma unroll
      for (int q = 0; q < V; ++q) s += a[j][q];
    }
  }
  s = warp_sum(s);
  const float mean = s / C;
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < NCH; ++j) {
    if (lane + 32 * j < nv) {
#pragma unroll
      for (int q = 0; q < V; ++q) { const float d = a[j][q] - mean; ss += d * d; }
    }
  }
  ss = warp_sum(ss);
  const float rstd = rsqrtf(ss / C + 1e-6f);
  const int b = (int)(r < seg_split ? r / rpb0 : (r - seg_split) / rpb1);
  // the block's sample from shared memory, a second sample (a block straddling
  // a sample boundary) from global memory
  const float* sh = b == b0 ? smod : shift + (size_t)b * mod_stride;
  const float* sc = b == b0 ? smod + C : scale + (size_t)b * mod_stride;
  T* orow = out + r * C;
#pragma unroll
  for (int j = 0; j < NCH; ++j) {
    const int k = lane + 32 * j;
    if (k < nv) {
      float o[V];
#pragma unroll
      for (int q = 0; q < V; q += 4) {
        const float4 s4 = *reinterpret_cast<const float4*>(sh + k * V + q);
        const float4 c4 = *reinterpret_cast<const float4*>(sc + k * V + q);
        o[q] = (a[j][q] - mean) * rstd * (1.0f + c4.x) + s4.x;
        o[q + 1] = (a[j][q + 1] - mean) * rstd * (1.0f + c4.y) + s4.y;
        o[q + 2] = (a[j][q + 2] - mean) * rstd * (1.0f + c4.z) + s4.z;
        o[q + 3] = (a[j][q + 3] - mean) * rstd * (1.0f + c4.w) + s4.w;
      }
      st16(orow + k * V, o);
    }
  }
}

// Each warp takes rpw rows (8 warps, a block of 8 * rpw consecutive rows);
// the block first stages the shift / scale vectors of its first row's
// sample in shared memory (coalesced, read back by every warp of that sample
// instead of 4 x 16 B per lane per chunk from global memory); a warp loads
// its next row while it reduces and writes the current one.
template <class T, int NCH>
__global__ void __launch_bounds__(256) k_ln_mod(const T* __restrict__ x, T* __restrict__ out, long long rows, int C,
                                                const float* __restrict__ shift, const float* __restrict__ scale,
                                                int mod_stride, int seg_split, int rpb0, int rpb1, int rpw) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float4 smod4[];                  // [2 * C / 4]: shift, then scale
  float* smod = reinterpret_cast<float*>(smod4);
  constexpr int V = VecN<T>::n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long r0 = (long long)blockIdx.x * 8 * rpw;
  const int b0 = (int)(r0 < seg_split ? r0 / rpb0 : (r0 - seg_split) / rpb1);
  const int nv = C / V;
  // rows r0 + warp * rpw + t, t < rpw; the first one's loads go out before
  // the staging
  const long long rw = r0 + (long long)warp * rpw;
  uint4 cur[NCH];
  auto load_row = [&](long long r, uint4 (&v)[NCH]) {
    const T* xr = x + r * C;
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
      const int k = lane + 32 * j;
      if (k < nv) v[j] = *reinterpret_cast<const uint4*>(xr + k * V);
    }
  };
  if (rw < rows) load_row(rw, cur);
  {
    const float4* sh4 = reinterpret_cast<const float4*>(shift + (size_t)b0 * mod_stride);
    const float4* sc4 = reinterpret_cast<const float4*>(scale + (size_t)b0 * mod_stride);
    for (int i = threadIdx.x; i < C / 4; i += blockDim.x) {
      smod4[i] = sh4[i];
      smod4[C / 4 + i] = sc4[i];
    }
  }
  __syncthreads();
  for (int t = 0; t < rpw; ++t) {
    const long long r = rw + t;
    if (r >= rows) break;
    uint4 nxt[NCH];
    const bool more = t + 1 < rpw && r + 1 < rows;
    if (more) load_row(r + 1, nxt);
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
      if (lane + 32 * j < nv) {
        float a[V];
        unpack16(cur[j], a);
#pragma unroll
        for (int q = 0; q < V; ++q) s += a[q];
      }
    }
    s = warp_sum(s);
    const float mean = s / C;
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
      if (lane + 32 * j < nv) {
        float a[V];
        unpack16(cur[j], a);
#pragma unroll
        for (int q = 0; q < V; ++q) { const float d = a[q] - mean; ss += d * d; }
      }
    }
    ss = warp_sum(ss);
    const float rstd = rsqrtf(ss / C + 1e-6f);
    const int b = (int)(r < seg_split ? r / rpb0 : (r - seg_split) / rpb1);
    // the block's sample from shared memory, another sample (a block
    // straddling a sample boundary) from global memory
    const float* sh = b == b0 ? smod : shift + (size_t)b * mod_stride;
    const float* sc = b == b0 ? smod + C : scale + (size_t)b * mod_stride;
    T* orow = out + r * C;
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
      const int k = lane + 32 * j;
      if (k < nv) {
        float a[V], o[V];
        unpack16(cur[j], a);
#pragma unroll
        for (int q = 0; q < V; q += 4) {
          const float4 s4 = *reinterpret_cast<const float4*>(sh + k * V + q);
          const float4 c4 = *reinterpret_cast<const float4*>(sc + k * V + q);
          o[q] = (a[q] - mean) * rstd * (1.0f + c4.x) + s4.x;
          o[q + 1] = (a[q + 1] - mean) * rstd * (1.0f + c4.y) + s4.y;
          o[q + 2] = (a[q + 2] - mean) * rstd * (1.0f + c4.z) + s4.z;
          o[q + 3] = (a[q + 3] - mean) * rstd * (1.0f + c4.w) + s4.w;
        }
        st16(orow + k * V, o);
      }
    }
    if (more) {
#pragma unroll
      for (int j = 0; j < NCH; ++j) cur[j] = nxt[j];
    }
  }
}

template <class T>
static cudaError_t ln_mod_t(const void* x, void* out, long long rows, int C, const float* shift, const float* scale,
                            int mod_stride, int seg_split, int rpb0, int rpb1, cudaStream_t s) {
  constexpr int V = VecN<T>::n;
  const int nch = (C / V + 31) / 32;
  // rows per warp: one while a row per warp makes at most about two waves
  // of blocks (every row's loads in flight at once), else enough that the
  // blocks fill about two per SM (measured: 4096 x 1152 rows 6.6 us with one
  // row per warp, 8.5 us with two; 14310 x 2048 rows 32.5 us with one, 24.5
  // us with six)
  const long long per_wave = 8LL * 2 * num_sms();
  int rpw = rows <= 2 * per_wave ? 1 : (int)((rows + per_wave - 1) / per_wave);
  rpw = rpw < 1 ? 1 : rpw > 8 ? 8 : rpw;
  const unsigned grid = (unsigned)((rows + 8LL * rpw - 1) / (8LL * rpw));
  const size_t smem = (size_t)2 * C * sizeof(float);  // shift + scale of one sample
  if (C % 4 != 0 || smem > 48 * 1024) return cudaErrorInvalidValue;
  const T* xp = (const T*)x;
  T* op = (T*)out;
#define FF_LN_CASE(n) \
  case n:                                                                                                              \
    if (rpw == 1)                                                                                                      \
      launch_pdl(k_ln_mod1<T, n>, grid, 256, smem, s, xp, op, rows, C, shift, scale, mod_stride, seg_split, rpb0, rpb1); \
    else                                                                                                               \
      launch_pdl(k_ln_mod<T, n>, grid, 256, smem, s, xp, op, rows, C, shift, scale, mod_stride, seg_split, rpb0, rpb1,  \
                 rpw);                                                                                                 \
    break;
  const int nchr = nch <= 6 ? nch : nch <= 8 ? 8 : nch <= 12 ? 12 : nch <= 16 ? 16 : 0;
  switch (nchr) {
    FF_LN_CASE(1) FF_LN_CASE(2) FF_LN_CASE(3) FF_LN_CASE(4) FF_LN_CASE(5) FF_LN_CASE(6)
    FF_LN_CASE(8) FF_LN_CASE(12) FF_LN_CASE(16)
    default:
      return cudaErrorInvalidValue;
  }
#undef FF_LN_CASE
  return launched();
}

cudaError_t launch_ln_mod(DType dt, const void* x, void* out, long long rows, int C, const float* shift,
                          const float* scale, int mod_stride, int seg_split, int rpb0, int rpb1, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (((uintptr_t)shift & 15) || ((uintptr_t)scale & 15) || (mod_stride & 3)) return cudaErrorInvalidValue;
  if (dt == F32) return ln_mod_t<float>(x, out, rows, C, shift, scale, mod_stride, seg_split, rpb0, rpb1, s);
  return ln_mod_t<bf16>(x, out, rows, C, shift, scale, mod_stride, seg_split, rpb0, rpb1, s);
}

// Sinusoidal features of every model time: row s = [cos(t_s f_k) | sin(t_s f_k)].
template <class T>
__global__ void k_sinusoid_table(const float* __restrict__ times, int S, T* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  const int s = blockIdx.x;
  if (s >= S) return;
  const double t = (double)times[s];
  for (int k = threadIdx.x; k < 128; k += blockDim.x) {
    const double f = exp(-log(10000.0) * (double)k / 128.0);
    out[(size_t)s * 256 + k] = from_f<T>((float)cos(t * f));
    out[(size_t)s * 256 + 128 + k] = from_f<T>((float)sin(t * f));
  }
}

cudaError_t launch_sinusoid_table(DType dt, const float* times, int S, void* out, cudaStream_t s) {
  if (S <= 0) return cudaSuccess;
  if (dt == F32) launch_pdl(k_sinusoid_table<float>, S, 128, 0, s, times, S, (float*)out);
  else launch_pdl(k_sinusoid_table<bf16>, S, 128, 0, s, times, S, (bf16*)out);
  return launched();
}

// SiLU(c) of every (step, sample): c = temb[step] (+ y_emb[label]).
template <class T>
__global__ void k_cond_table(const float* __restrict__ temb, const T* __restrict__ y_emb, const int* __restrict__ labels,
                             int S, int B, int C, const int* __restrict__ need_row, T* __restrict__ all,
                             T* __restrict__ need) {
  pdl_trigger();
  pdl_wait();
  const int row = blockIdx.x;  // s * B + b
  const int s = row / B, b = row % B;
  if (s >= S) return;
  const int nr = need_row ? need_row[s] : -1;
  for (int k = threadIdx.x; k < C; k += blockDim.x) {
    float v = temb[(size_t)s * C + k];
    if (y_emb) v += to_f(y_emb[(size_t)labels[b] * C + k]);
    const T o = from_f<T>(silu(v));
    all[(size_t)row * C + k] = o;
    if (nr >= 0) need[((size_t)nr * B + b) * C + k] = o;
  }
}

cudaError_t launch_cond_table(DType dt, const float* temb, const void* y_emb, const int* labels, int S, int B, int C,
                              const int* need_row, void* all, void* need, cudaStream_t s) {
  if (S <= 0) return cudaSuccess;
  if (dt == F32)
    launch_pdl(k_cond_table<float>, S * B, 256, 0, s, temb, (const float*)y_emb, labels, S, B, C, need_row, (float*)all,
                                              (float*)need);
  else
    launch_pdl(k_cond_table<bf16>, S * B, 256, 0, s, temb, (const bf16*)y_emb, labels, S, B, C, need_row, (bf16*)all,
                                             (bf16*)need);
  return launched();
}

// Patch features of the model batch (latent sample b % B_lat): row
// b*N_img + token, feature (channel, frame offset, row offset, col offset).
template <class T>
__global__ void k_patchify(const float* __restrict__ lat, int B_lat, int B_model, int Cin, int F, int H, int W, int p,
                           int pt, T* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  const int Ff = F > 0 ? F : 1, ptt = F > 0 ? pt : 1;
  const int gf = Ff / ptt, gh = H / p, gw = W / p;
  const int P = ptt * p * p, feat = Cin * P;
  const long long total = (long long)B_model * gf * gh * gw * feat;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long long)gridDim.x * blockDim.x) {
    const int f = (int)(i % feat);
    const long long row = i / feat;
    const int tok = (int)(row % ((long long)gf * gh * gw));
    const int b = (int)(row / ((long long)gf * gh * gw));
    const int c = f / P, o = f % P;
    const int ot = o / (p * p), oh = (o / p) % p, ow = o % p;
    const int tw = tok % gw, th = (tok / gw) % gh, tf = tok / (gw * gh);
    const int zf = tf * ptt + ot, zh = th * p + oh, zw = tw * p + ow;
    const long long src = ((((long long)(b % B_lat) * Cin + c) * Ff + zf) * H + zh) * W + zw;
    out[i] = from_f<T>(lat[src]);
  }
}

cudaError_t launch_patchify(DType dt, const float* latent, int B_lat, int B_model, int Cin, int F, int H, int W,
                            int p, int pt, void* out, cudaStream_t s) {
  const int grid = num_sms() * 4;
  if (dt == F32) launch_pdl(k_patchify<float>, grid, 256, 0, s, latent, B_lat, B_model, Cin, F, H, W, p, pt, (float*)out);
  else launch_pdl(k_patchify<bf16>, grid, 256, 0, s, latent, B_lat, B_model, Cin, F, H, W, p, pt, (bf16*)out);
  return launched();
}

template <class T>
__global__ void k_convert(const float* __restrict__ in, T* __restrict__ out, long long n) {
  pdl_trigger();
  pdl_wait();
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
    out[i] = from_f<T>(in[i]);
}

cudaError_t launch_convert(DType dt, const float* in, void* out, long long n, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int grid = num_sms() * 4;
  if (dt == F32) launch_pdl(k_convert<float>, grid, 256, 0, s, in, (float*)out, n);
  else launch_pdl(k_convert<bf16>, grid, 256, 0, s, in, (bf16*)out, n);
  return launched();
}

// Guidance + sampler update of the latent: g = out_u + s (out_c - out_u)
// (or out), x <- c1 x + c2 g, reading the model output through the
// unpatchify index map.  Euler: c1 = 1, c2 = sigma_{i+1} - sigma_i.  DDIM:
// c1 = sqrt(a_prev / a_t), c2 = sqrt(1 - a_prev) - sqrt(a_prev (1 - a_t) / a_t).
__global__ void k_sampler(const float* __restrict__ mo, float* __restrict__ lat, int B_lat, int cfg, float cfg_scale,
                          int Cin, int Cout, int F, int H, int W, int p, int pt, float c1, float c2) {
  pdl_trigger();
  pdl_wait();
  const int Ff = F > 0 ? F : 1, ptt = F > 0 ? pt : 1;
  const int gh = H / p, gw = W / p, gf = Ff / ptt;
  const int P = ptt * p * p;
  const long long ntok = (long long)gf * gh * gw;
  const long long total = (long long)B_lat * Cin * Ff * H * W;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long long)gridDim.x * blockDim.x) {
    const int zw = (int)(i % W);
    const int zh = (int)((i / W) % H);
    const int zf = (int)((i / ((long long)W * H)) % Ff);
    const int c = (int)((i / ((long long)W * H * Ff)) % Cin);
    const int b = (int)(i / ((long long)W * H * Ff * Cin));
    const long long tok = ((long long)(zf / ptt) * gh + zh / p) * gw + zw / p;
    const int f = c * P + ((zf % ptt) * p + zh % p) * p + zw % p;
    const long long fo = (long long)Cout * P;
    float g = mo[((long long)b * ntok + tok) * fo + f];
    if (cfg) {
      const float gu = mo[((long long)(b + B_lat) * ntok + tok) * fo + f];
      g = gu + cfg_scale * (g - gu);
    }
    lat[i] = c1 * lat[i] + c2 * g;
  }
}

cudaError_t launch_sampler(const float* model_out, float* latent, int B_lat, int cfg, float cfg_scale, int Cin,
                           int Cout, int F, int H, int W, int p, int pt, float c1, float c2, cudaStream_t s) {
  launch_pdl(k_sampler, num_sms() * 2, 256, 0, s, model_out, latent, B_lat, cfg, cfg_scale, Cin, Cout, F, H, W, p, pt, c1, c2);
  return launched();
}

// Seeded N(0,1) latent: SplitMix64 word k = mix(seed + (k+1) * golden),
// u = ((w >> 11) + 0.5) 2^-53, Box-Muller on word pairs (2m, 2m+1).
__device__ __forceinline__ unsigned long long splitmix_word(unsigned long long seed, unsigned long long k) {
  unsigned long long z = seed + (k + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__global__ void k_noise(unsigned long long seed, float* __restrict__ out, long long n) {
  pdl_trigger();
  pdl_wait();
  const long long pairs = (n + 1) / 2;
  for (long long m = (long long)blockIdx.x * blockDim.x + threadIdx.x; m < pairs; m += (long long)gridDim.x * blockDim.x) {
    const double u1 = ((double)(splitmix_word(seed, 2 * m) >> 11) + 0.5) * 0x1.0p-53;
    const double u2 = ((double)(splitmix_word(seed, 2 * m + 1) >> 11) + 0.5) * 0x1.0p-53;
    const double r = sqrt(-2.0 * log(u1));
    double sn, cs;
    sincos(2.0 * 3.141592653589793 * u2, &sn, &cs);
    out[2 * m] = (float)(r * cs);
    if (2 * m + 1 < n) out[2 * m + 1] = (float)(r * sn);
  }
}

cudaError_t launch_noise(unsigned long long seed, float* out, long long n, cudaStream_t s) {
  launch_pdl(k_noise, num_sms() * 2, 256, 0, s, seed, out, n);
  return launched();
}

// Fixed 2-D sin-cos position embedding replicated over B samples:
// channels [0, C/2) encode the patch row, [C/2, C) the column, each half
// [sin(pos w_k) | cos(pos w_k)], w_k = 10000^(-k/(C/4)).
template <class T>
__global__ void k_pos2d(T* __restrict__ out, int B, int gh, int gw, int C) {
  pdl_trigger();
  pdl_wait();
  const int q = C / 4;
  const long long total = (long long)B * gh * gw * C;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long long)gridDim.x * blockDim.x) {
    const int c = (int)(i % C);
    const int tok = (int)((i / C) % ((long long)gh * gw));
    const int half = c / (C / 2), cc = c % (C / 2);
    const double pos = half == 0 ? (double)(tok / gw) : (double)(tok % gw);
    const int k = cc % q;
    const double a = pos * pow(10000.0, -(double)k / (double)q);
    out[i] = from_f<T>((float)(cc < q ? sin(a) : cos(a)));
  }
}

cudaError_t launch_pos2d(DType dt, void* out, int B, int gh, int gw, int C, cudaStream_t s) {
  const int grid = num_sms() * 4;
  if (dt == F32) launch_pdl(k_pos2d<float>, grid, 256, 0, s, (float*)out, B, gh, gw, C);
  else launch_pdl(k_pos2d<bf16>, grid, 256, 0, s, (bf16*)out, B, gh, gw, C);
  return launched();
}

}  // namespace ff
