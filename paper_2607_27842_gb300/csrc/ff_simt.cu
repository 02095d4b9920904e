// CUDA-core (no tensor core, no TF32) dense layer and attention: the fp32
// mode of the exact block (Eq. 1) and the narrow final projection.
#include "ff_common.cuh"

#include <math.h>

namespace ff {

// ---------------------------------------------------------------------------
// out = epilogue(A[M,K] W[N,K]^T), 64 x 128 tile, BK = 16, each thread owns
// 4 rows x 8 consecutive columns.  Operands are converted to fp32 in shared
// memory; accumulation is fp32 FFMA.
// ---------------------------------------------------------------------------
constexpr int SG_BM = 64, SG_BN = 128, SG_BK = 16;

template <class T>
__global__ void __launch_bounds__(256) k_gemm_simt(int M, int N, int K, const T* __restrict__ A, int lda,
                                                   const T* __restrict__ W, int ldw, EpiArgs e) {
  __shared__ __align__(16) float As[SG_BK][SG_BM + 4];
  __shared__ __align__(16) float Ws[SG_BK][SG_BN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int m0 = blockIdx.y * SG_BM, n0 = blockIdx.x * SG_BN;
  float acc[4][8];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < K; k0 += SG_BK) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int idx = threadIdx.x + q * 256;  // 0 .. 1023 over [64 rows][16 k]
      const int r = idx >> 4, kk = idx & 15;
      const int gm = m0 + r, gk = k0 + kk;
      As[kk][r] = (gm < M && gk < K) ? to_f(A[(size_t)gm * lda + gk]) : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int idx = threadIdx.x + q * 256;  // 0 .. 2047 over [128 rows][16 k]
      const int r = idx >> 4, kk = idx & 15;
      const int gn = n0 + r, gk = k0 + kk;
      Ws[kk][r] = (gn < N && gk < K) ? to_f(W[(size_t)gn * ldw + gk]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < SG_BK; ++kk) {
      const float4 a4 = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
      const float4 b0 = *reinterpret_cast<const float4*>(&Ws[kk][tx * 8]);
      const float4 b1 = *reinterpret_cast<const float4*>(&Ws[kk][tx * 8 + 4]);
      const float a[4] = {a4.x, a4.y, a4.z, a4.w};
      const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  const int nc = n0 + tx * 8;
  if (nc >= N) return;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m < M) epi_chunk<T, 8>(e, m, nc, N, acc[i]);
  }
}

cudaError_t gemm_simt(DType dt, int M, int N, int K, const void* A, int lda, const void* W, int ldw,
                      const EpiArgs& e, cudaStream_t s) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  dim3 grid((N + SG_BN - 1) / SG_BN, (M + SG_BM - 1) / SG_BM);
  if (dt == F32)
    k_gemm_simt<float><<<grid, 256, 0, s>>>(M, N, K, (const float*)A, lda, (const float*)W, ldw, e);
  else
    k_gemm_simt<bf16><<<grid, 256, 0, s>>>(M, N, K, (const bf16*)A, lda, (const bf16*)W, ldw, e);
  return launched();
}

// ---------------------------------------------------------------------------
// Attention on CUDA cores: one warp per query row, keys in chunks of 32
// (lane j scores key j of the chunk), online softmax, each lane owns output
// dims lane, lane + 32, ... (d <= 128).
// ---------------------------------------------------------------------------
__device__ __forceinline__ long long tok_row(const AttnArgs& a, int b, int n) {
  return n < a.Nt ? (long long)b * a.Nt + n : (long long)a.B * a.Nt + (long long)b * a.Ni + (n - a.Nt);
}

template <class T>
__global__ void __launch_bounds__(256) k_attn_simt(AttnArgs a, float scale) {
  __shared__ float qs[8][128];
  const int N = a.Nt + a.Ni;
  const int h = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qi = blockIdx.x * 8 + warp;
  if (qi >= N) return;
  const T* Q = reinterpret_cast<const T*>(a.q);
  const T* Kp = reinterpret_cast<const T*>(a.k);
  const T* Vp = reinterpret_cast<const T*>(a.v);
  const long long qr = tok_row(a, b, qi);
  for (int e = lane; e < a.hd; e += 32) qs[warp][e] = to_f(Q[qr * a.ld_qkv + (size_t)h * a.hd + e]);
  __syncwarp();
  float m = -INFINITY, l = 0.f, o[4] = {0.f, 0.f, 0.f, 0.f};
  for (int c0 = 0; c0 < N; c0 += 32) {
    const int key = c0 + lane;
    float sc = -INFINITY;
    if (key < N) {
      const T* kr = Kp + tok_row(a, b, key) * a.ld_qkv + (size_t)h * a.hd;
      float dot = 0.f;
      for (int e = 0; e < a.hd; ++e) dot = fmaf(qs[warp][e], to_f(kr[e]), dot);
      sc = dot * scale;
    }
    float cmax = sc;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) cmax = fmaxf(cmax, __shfl_xor_sync(0xffffffffu, cmax, off));
    const float mn = fmaxf(m, cmax);
    const float alpha = expf(m - mn);
    const float p = key < N ? expf(sc - mn) : 0.f;
    float psum = p;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, off);
    l = l * alpha + psum;
#pragma unroll
    for (int j = 0; j < 4; ++j) o[j] *= alpha;
    const int nk = min(32, N - c0);
    for (int j = 0; j < nk; ++j) {
      const float pj = __shfl_sync(0xffffffffu, p, j);
      const T* vr = Vp + tok_row(a, b, c0 + j) * a.ld_qkv + (size_t)h * a.hd;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int e = lane + 32 * q;
        if (e < a.hd) o[q] = fmaf(pj, to_f(vr[e]), o[q]);
      }
    }
    m = mn;
  }
  T* out = reinterpret_cast<T*>(a.out) + qr * a.ld_out + (size_t)h * a.hd;
  const float inv = 1.0f / l;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int e = lane + 32 * q;
    if (e < a.hd) out[e] = from_f<T>(o[q] * inv);
  }
}

cudaError_t attention_simt(DType dt, const AttnArgs& a, cudaStream_t s) {
  const int N = a.Nt + a.Ni;
  dim3 grid((N + 7) / 8, a.H, a.B);
  const float scale = 1.0f / sqrtf((float)a.hd);
  if (dt == F32) k_attn_simt<float><<<grid, 256, 0, s>>>(a, scale);
  else k_attn_simt<bf16><<<grid, 256, 0, s>>>(a, scale);
  return launched();
}

}  // namespace ff
