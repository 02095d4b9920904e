// Non-causal multi-head attention inside the exact block (Eq. 1) over the
// joint [text ; image] token sequence of each sample.  bf16 runs on the
// tcgen05 kernel of ff_attention_tc.cu when the fused qkv layout allows;
// otherwise (and for head widths 32):
//
// bf16: flash-style kernel on warp-level mma.sync (m16n8k16, fp32
// accumulate): 64 queries per CTA (16 per warp), keys/values streamed in
// 64-row tiles through a double-buffered cp.async ring, online softmax in
// registers, P re-packed from the score accumulators as the A operand of
// P V.  Head widths that are not a multiple of 16 (72) are zero-padded in
// shared memory for q k^T only.
#include "ff_common.cuh"

#include <math.h>

namespace ff {

namespace {

__device__ __forceinline__ uint32_t saddr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void cp_async16(void* dst, const void* src, int bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(saddr(dst)), "l"(src), "r"(bytes) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(saddr(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(saddr(p)));
}
__device__ __forceinline__ void ldsm_x2_t(uint32_t (&r)[2], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0, %1}, [%2];"
               : "=r"(r[0]), "=r"(r[1])
               : "r"(saddr(p)));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ long long row_of(const AttnArgs& a, int b, int n) {
  return n < a.Nt ? (long long)b * a.Nt + n : (long long)a.B * a.Nt + (long long)b * a.Ni + (n - a.Nt);
}

constexpr int BQ = 64, BKV = 64;

template <int D> struct AttCfg {
  static constexpr int DK = (D + 15) / 16 * 16;  // q k^T reduction width (zero padded)
  static constexpr int NTD = D / 8;              // 8-wide output column tiles
  static constexpr int LDS = DK + 8;             // smem row stride: ldmatrix rows hit distinct banks
  static constexpr int CPR = D / 8;              // 16-byte chunks per head row
  static constexpr size_t SMEM = (size_t)(BQ + 4 * BKV) * LDS * sizeof(bf16);
};

template <int D>
__global__ void __launch_bounds__(128) k_attn_mma(AttnArgs a, float scale_log2) {
  using Cf = AttCfg<D>;
  constexpr int DK = Cf::DK, NTD = Cf::NTD, LDS = Cf::LDS, CPR = Cf::CPR;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  bf16* sQ = reinterpret_cast<bf16*>(smem_raw);
  bf16* sK = sQ + BQ * LDS;
  bf16* sV = sK + 2 * BKV * LDS;

  const int N = a.Nt + a.Ni;
  const int q0 = blockIdx.x * BQ, h = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bf16* Qg = reinterpret_cast<const bf16*>(a.q);
  const bf16* Kg = reinterpret_cast<const bf16*>(a.k);
  const bf16* Vg = reinterpret_cast<const bf16*>(a.v);
  const size_t hoff = (size_t)h * D;

  if constexpr (DK > D) {  // zero the reduction padding of Q and both K buffers
    constexpr int PADW = DK > D ? DK - D : 1;
    for (int i = tid; i < (BQ + 2 * BKV) * PADW; i += 128) {
      const int r = i / PADW, c = D + i % PADW;
      bf16* base = r < BQ ? sQ + r * LDS : sK + (r - BQ) * LDS;
      base[c] = __float2bfloat16_rn(0.f);
    }
  }
  for (int c = tid; c < BQ * CPR; c += 128) {
    const int r = c / CPR, j = c % CPR;
    const int n = q0 + r;
    const bool ok = n < N;
    const bf16* src = ok ? Qg + row_of(a, b, n) * a.ld_qkv + hoff + j * 8 : Qg;
    cp_async16(sQ + r * LDS + j * 8, src, ok ? 16 : 0);
  }
  auto load_kv = [&](int blk, int buf) {
    bf16* dk = sK + buf * BKV * LDS;
    bf16* dv = sV + buf * BKV * LDS;
    for (int c = tid; c < BKV * CPR; c += 128) {
      const int r = c / CPR, j = c % CPR;
      const int n = blk * BKV + r;
      const bool ok = n < N;
      const long long row = ok ? row_of(a, b, n) : 0;
      cp_async16(dk + r * LDS + j * 8, ok ? Kg + row * a.ld_qkv + hoff + j * 8 : Kg, ok ? 16 : 0);
      cp_async16(dv + r * LDS + j * 8, ok ? Vg + row * a.ld_qkv + hoff + j * 8 : Vg, ok ? 16 : 0);
    }
  };
  load_kv(0, 0);
  cp_commit();
  cp_wait_all();
  __syncthreads();

  uint32_t qf[DK / 16][4];
#pragma unroll
  for (int kk = 0; kk < DK / 16; ++kk) {
    const int r = warp * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
    const int c = kk * 16 + ((lane >> 4) << 3);
    ldsm_x4(qf[kk], sQ + r * LDS + c);
  }

  float o[NTD][4];
#pragma unroll
  for (int i = 0; i < NTD; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  const int g = lane >> 2, t = lane & 3;
  const int nkv = (N + BKV - 1) / BKV;

  for (int j = 0; j < nkv; ++j) {
    const int buf = j & 1;
    if (j + 1 < nkv) {
      load_kv(j + 1, buf ^ 1);
      cp_commit();
    }
    const bf16* cK = sK + buf * BKV * LDS;
    const bf16* cV = sV + buf * BKV * LDS;
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < DK / 16; ++kk) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t r[4];
        const int kr = np * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int kc = kk * 16 + (((lane >> 3) & 1) << 3);
        ldsm_x4(r, cK + kr * LDS + kc);
        mma16816(s[2 * np], qf[kk], r[0], r[1]);
        mma16816(s[2 * np + 1], qf[kk], r[2], r[3]);
      }
    }
    const bool ragged = (j + 1) * BKV > N;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float v = s[nt][e] * scale_log2;
        if (ragged && j * BKV + nt * 8 + 2 * t + (e & 1) >= N) v = -INFINITY;
        s[nt][e] = v;
      }
    }
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      mx[0] = fmaxf(mx[0], fmaxf(s[nt][0], s[nt][1]));
      mx[1] = fmaxf(mx[1], fmaxf(s[nt][2], s[nt][3]));
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
    }
    float alpha[2], psum[2] = {0.f, 0.f};
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const float mn = fmaxf(mrow[r], mx[r]);
      alpha[r] = exp2f(mrow[r] - mn);
      mrow[r] = mn;
    }
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float p = exp2f(s[nt][e] - mrow[e >> 1]);
        s[nt][e] = p;
        psum[e >> 1] += p;
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) lrow[r] = lrow[r] * alpha[r] + psum[r];
#pragma unroll
    for (int i = 0; i < NTD; ++i) {
      o[i][0] *= alpha[0]; o[i][1] *= alpha[0];
      o[i][2] *= alpha[1]; o[i][3] *= alpha[1];
    }
#pragma unroll
    for (int kk = 0; kk < BKV / 16; ++kk) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      pa[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      pa[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      pa[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
      const int vr = kk * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
#pragma unroll
      for (int dp = 0; dp < NTD / 2; ++dp) {
        uint32_t r[4];
        ldsm_x4_t(r, cV + vr * LDS + dp * 16 + ((lane >> 4) << 3));
        mma16816(o[2 * dp], pa, r[0], r[1]);
        mma16816(o[2 * dp + 1], pa, r[2], r[3]);
      }
      if (NTD & 1) {
        uint32_t r[2];
        ldsm_x2_t(r, cV + vr * LDS + (NTD - 1) * 8);
        mma16816(o[NTD - 1], pa, r[0], r[1]);
      }
    }
    cp_wait_all();
    __syncthreads();
  }

#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
  }
  bf16* Og = reinterpret_cast<bf16*>(a.out);
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int n = q0 + warp * 16 + g + 8 * r;
    if (n >= N) continue;
    const float inv = 1.0f / lrow[r];
    bf16* orow = Og + row_of(a, b, n) * a.ld_out + hoff;
#pragma unroll
    for (int i = 0; i < NTD; ++i) {
      __nv_bfloat162 v = __floats2bfloat162_rn(o[i][2 * r] * inv, o[i][2 * r + 1] * inv);
      *reinterpret_cast<__nv_bfloat162*>(orow + i * 8 + 2 * t) = v;
    }
  }
}

template <int D>
cudaError_t attn_mma_t(const AttnArgs& a, cudaStream_t s) {
  const size_t smem = AttCfg<D>::SMEM;
  cudaError_t e = cudaFuncSetAttribute(k_attn_mma<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int N = a.Nt + a.Ni;
  dim3 grid((N + BQ - 1) / BQ, a.H, a.B);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)D);
  k_attn_mma<D><<<grid, 128, smem, s>>>(a, scale_log2);
  return launched();
}

}  // namespace

cudaError_t attention(DType dt, const AttnArgs& a, cudaStream_t s) {
  if (a.B <= 0 || a.H <= 0 || a.Nt + a.Ni <= 0) return cudaSuccess;
  if (dt == BF16) {
    // tensor cores (tcgen05) whenever the layout allows
    const cudaError_t e = attention_tc(a, s);
    if (e != cudaErrorInvalidValue && e != cudaErrorNotSupported) return e;
    switch (a.hd) {
      case 32: return attn_mma_t<32>(a, s);
      case 64: return attn_mma_t<64>(a, s);
      case 72: return attn_mma_t<72>(a, s);
      case 128: return attn_mma_t<128>(a, s);
      default: break;
    }
  }
  return attention_simt(dt, a, s);
}

}  // namespace ff
