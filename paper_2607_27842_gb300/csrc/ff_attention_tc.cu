// Non-causal attention softmax(q k^T / sqrt(d)) v of the exact block (Eq. 1)
// on the 5th-generation tensor cores, bf16 in, fp32 accumulate.
//
// One CTA per (sample, head, 128-query tile), 6 warps:
//   warp 0     TMA producer: the query tile once, key / value tiles of 128
//              tokens into a 2-stage ring, straight from the fused qkv
//              activation (3-D tensor map: head width, head slot, row; the
//              head width is zero-padded to a multiple of 64 by the map);
//   warp 1     TMEM allocator and MMA issuer: S = Q K^T into one of two TMEM
//              score buffers (tcgen05.mma, both operands K-major), then
//              O += P V into the TMEM output accumulator (P K-major from
//              shared memory, V MN-major straight from its tile);
//   warps 2-5  softmax: each thread owns one query row (its TMEM lane):
//              row max, exp2, row sum, P written as bf16 into shared memory
//              in the 128-byte-swizzled operand layout; the output row is
//              rescaled in TMEM only when the running max grew by more than
//              2^8 (the normalisation divides by the same stale max).
// Keys of a sample lie in up to two row segments (text rows, image rows of
// the stream-major token layout); tiles never straddle a segment and keys
// past a segment's end are masked.
#include "ff_common.cuh"
#include "ff_tc.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <math.h>
#include <mutex>

namespace ff {

namespace {

using namespace tc;

constexpr int AQ = 128;        // queries per CTA (MMA M)
constexpr int AKV = 128;       // keys per tile (MMA N of S, K of P V)
constexpr int ATHREADS = 192;
constexpr int KV_STAGES = 2;
constexpr float RESCALE_LOG2 = 8.0f;

__device__ unsigned int g_attn_watchdog;

__device__ __forceinline__ bool wait_a(uint64_t* b, uint32_t parity, volatile int* abort_flag) {
  return mbar_wait(b, parity, abort_flag, &g_attn_watchdog);
}

template <int D> struct ACfg {
  static constexpr int NBOX = D <= 64 ? 1 : 2;           // 64-wide column boxes per tile row
  static constexpr int DK = (D + 15) / 16 * 16;          // q k^T reduction width and P V output width
  static constexpr uint32_t BOX = 128 * 128;             // one [128 rows x 64] bf16 box, 16 KB
  static constexpr uint32_t Q_BYTES = NBOX * BOX;
  static constexpr uint32_t P_BYTES = 2 * BOX;           // [128 queries x 128 keys] bf16
  static constexpr uint32_t KV_BYTES = 2 * NBOX * BOX;   // K tile + V tile
  static constexpr size_t SMEM = 1024 + Q_BYTES + P_BYTES + (size_t)KV_STAGES * KV_BYTES + 256;
  static constexpr uint32_t TMEM_O = 2 * AKV;            // columns [0,256) scores x2, then O
  // kind::f16, D fp32, A/B bf16; S: both K-major, N = 128; O: B (V) MN-major (bit 16), N = DK
  static constexpr uint32_t IDESC_S = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(AKV >> 3) << 17) |
                                      ((uint32_t)(AQ >> 4) << 24);
  static constexpr uint32_t IDESC_O = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) | ((uint32_t)(DK >> 3) << 17) |
                                      ((uint32_t)(AQ >> 4) << 24);
};

// MN-major operand with 128-byte swizzle: 64 contiguous elements (128 B) per
// row of the swizzle atom, 8 rows 128 B apart along K; the next 64-element
// group along MN sits `lbo` bytes further, the next 8-row group along K
// 1024 B further.
__device__ __forceinline__ uint64_t sw128_desc_mn(uint32_t addr, uint32_t lbo) {
  uint64_t d = (uint64_t)((addr & 0x3FFFF) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

__device__ __forceinline__ void tma_load3(const CUtensorMap* tm, uint64_t* bar, void* dst, int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];" ::"r"(saddr(dst)),
      "l"((uint64_t)tm), "r"(x), "r"(y), "r"(z), "r"(saddr(bar))
      : "memory");
}

// Row segments of sample b: text rows [b*Nt, b*Nt + Nt), image rows
// [B*Nt + b*Ni, ... + Ni).  Tile t of the sample's sequence: first row and
// number of valid rows.
struct SegTile {
  int row0, valid;
};
__device__ __forceinline__ SegTile seg_tile(const AttnArgs& a, int b, int t) {
  const int nt_tiles = (a.Nt + 127) / 128;
  if (t < nt_tiles) return {b * a.Nt + t * 128, min(128, a.Nt - t * 128)};
  const int u = t - nt_tiles;
  return {a.B * a.Nt + b * a.Ni + u * 128, min(128, a.Ni - u * 128)};
}

template <int D>
__global__ void __launch_bounds__(ATHREADS, 1)
    k_attn_tc(const __grid_constant__ CUtensorMap tmQKV, AttnArgs a, float scale_log2) {
  using C = ACfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;
  uint8_t* sP = sQ + C::Q_BYTES;
  uint8_t* sKV = sP + C::P_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sKV + KV_STAGES * C::KV_BYTES);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;
  uint64_t* kv_empty = kv_full + KV_STAGES;
  uint64_t* s_full = kv_empty + KV_STAGES;
  uint64_t* p_ready = s_full + 2;
  uint64_t* o_done = p_ready + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(o_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int nkv = (a.Nt + 127) / 128 + (a.Ni + 127) / 128;
  const SegTile qs = seg_tile(a, b, qt);

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < KV_STAGES; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_ready[i], 128);
    }
    mbar_init(o_done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmQKV) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(tmem_slot)), "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // query tile: head slot h
      mbar_expect_tx(q_full, C::Q_BYTES);
      for (int bx = 0; bx < C::NBOX; ++bx) tma_load3(&tmQKV, q_full, sQ + bx * C::BOX, 64 * bx, h, qs.row0);
      for (int j = 0; j < nkv; ++j) {
        const int s = j % KV_STAGES;
        const uint32_t ph = (j / KV_STAGES) & 1;
        if (!wait_a(&kv_empty[s], ph ^ 1, abort_flag)) break;
        const SegTile ks = seg_tile(a, b, j);
        uint8_t* kdst = sKV + s * C::KV_BYTES;
        uint8_t* vdst = kdst + C::NBOX * C::BOX;
        mbar_expect_tx(&kv_full[s], C::KV_BYTES);
        for (int bx = 0; bx < C::NBOX; ++bx) {
          tma_load3(&tmQKV, &kv_full[s], kdst + bx * C::BOX, 64 * bx, a.H + h, ks.row0);
          tma_load3(&tmQKV, &kv_full[s], vdst + bx * C::BOX, 64 * bx, 2 * a.H + h, ks.row0);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = wait_a(q_full, 0, abort_flag);
      const uint64_t qd = sw128_desc(saddr(sQ));
      const uint64_t pd = sw128_desc(saddr(sP));
      for (int j = 0; j <= nkv && ok; ++j) {
        if (j < nkv) {  // S_j = Q K_j^T into score buffer j % 2
          const int s = j % KV_STAGES;
          if (!wait_a(&kv_full[s], (j / KV_STAGES) & 1, abort_flag)) break;
          tc_fence_after();
          const uint64_t kd = sw128_desc(saddr(sKV + s * C::KV_BYTES));
#pragma unroll
          for (int k = 0; k < C::DK / 16; ++k) {
            // 16-wide k step k: box k / 4, +32 B per step inside the box
            const uint64_t off = (uint64_t)((k >> 2) * (C::BOX >> 4) + 2 * (k & 3));
            umma(tmem + (uint32_t)((j & 1) * AKV), qd + off, kd + off, C::IDESC_S, k != 0);
          }
          umma_commit(&s_full[j & 1]);
        }
        if (j >= 1) {  // O += P_{j-1} V_{j-1}
          const int jp = j - 1, s = jp % KV_STAGES;
          if (!wait_a(&p_ready[jp & 1], (jp >> 1) & 1, abort_flag)) break;
          tc_fence_after();
          const uint32_t vaddr = saddr(sKV + s * C::KV_BYTES + C::NBOX * C::BOX);
#pragma unroll
          for (int k = 0; k < AKV / 16; ++k) {
            // P: K-major, keys 64 per box; V: MN-major, 16 keys = 2 groups of 8 rows (2 KB)
            const uint64_t poff = (uint64_t)((k >> 2) * (C::BOX >> 4) + 2 * (k & 3));
            const uint64_t vd = sw128_desc_mn(vaddr + (uint32_t)k * 2048u, C::BOX);
            umma(tmem + C::TMEM_O, pd + poff, vd, C::IDESC_O, (jp | k) != 0);
          }
          umma_commit(o_done);
          umma_commit(&kv_empty[s]);
        }
      }
    }
  } else {
    // softmax: row r of the tile = TMEM lane r
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkv && ok; ++j) {
      const SegTile ks = seg_tile(a, b, j);
      int w = 1;
      if (lane == 0) w = wait_a(&s_full[j & 1], (j >> 1) & 1, abort_flag) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
      tc_fence_after();
      const uint32_t sbase = lane_base + (uint32_t)((j & 1) * AKV);
      float mx = -INFINITY;
#pragma unroll
      for (int c = 0; c < AKV / 32; ++c) {
        float v[32];
        tmem_ld32(sbase + (uint32_t)(c * 32), v);
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (c * 32 + e < ks.valid) mx = fmaxf(mx, v[e] * scale_log2);
      }
      const float m_new = fmaxf(m, mx);
      const bool grow = m_new > m + RESCALE_LOG2;  // also true on the first tile
      const float m_use = grow ? m_new : m;
      const float alpha = grow ? exp2f(m - m_new) : 1.0f;
      if (j >= 1) {  // O and the P buffer are free once P_{j-1} V_{j-1} completed
        int w2 = 1;
        if (lane == 0) w2 = wait_a(o_done, (j - 1) & 1, abort_flag) ? 1 : 0;
        if (!__shfl_sync(0xffffffffu, w2, 0)) { ok = false; break; }
        tc_fence_after();
        if (__any_sync(0xffffffffu, grow)) {
#pragma unroll
          for (int c = 0; c < C::DK / 16; ++c) {
            float o[16];
            tmem_ld16(lane_base + C::TMEM_O + (uint32_t)(c * 16), o);
#pragma unroll
            for (int e = 0; e < 16; ++e) o[e] *= alpha;
            tmem_st16(lane_base + C::TMEM_O + (uint32_t)(c * 16), o);
          }
        }
      }
      l *= alpha;
      m = m_use;
      // P row: 128 keys as bf16, 16-byte chunks swizzled by row (128B swizzle)
#pragma unroll
      for (int c = 0; c < AKV / 32; ++c) {
        float v[32];
        tmem_ld32(sbase + (uint32_t)(c * 32), v);
        uint32_t pk[16];
#pragma unroll
        for (int e = 0; e < 32; e += 2) {
          const float p0 = (c * 32 + e < ks.valid) ? exp2f(v[e] * scale_log2 - m) : 0.f;
          const float p1 = (c * 32 + e + 1 < ks.valid) ? exp2f(v[e + 1] * scale_log2 - m) : 0.f;
          l += p0 + p1;
          __nv_bfloat162 t = __floats2bfloat162_rn(p0, p1);
          pk[e >> 1] = *reinterpret_cast<uint32_t*>(&t);
        }
        // keys c*32 .. c*32+31: box (c >> 1), 16-byte chunks 4*(c & 1) .. +3
        uint8_t* rowp = sP + (c >> 1) * C::BOX + r * 128;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int chunk = 4 * (c & 1) + k;
          *reinterpret_cast<uint4*>(rowp + ((chunk ^ (r & 7)) << 4)) =
              make_uint4(pk[4 * k], pk[4 * k + 1], pk[4 * k + 2], pk[4 * k + 3]);
        }
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      tc_fence_before();
      mbar_arrive(&p_ready[j & 1]);
    }
    if (ok) {
      int w = 1;
      if (lane == 0) w = wait_a(o_done, (nkv - 1) & 1, abort_flag) ? 1 : 0;
      if (__shfl_sync(0xffffffffu, w, 0)) {
        tc_fence_after();
        const float inv = 1.0f / l;
        bf16* orow = reinterpret_cast<bf16*>(a.out) + (size_t)(qs.row0 + r) * a.ld_out + (size_t)h * D;
#pragma unroll
        for (int c = 0; c < C::DK / 16; ++c) {
          float o[16];
          tmem_ld16(lane_base + C::TMEM_O + (uint32_t)(c * 16), o);
          if (r < qs.valid) {
#pragma unroll
            for (int e = 0; e < 16; e += 8) {
              if (c * 16 + e < D) {
                float t[8];
#pragma unroll
                for (int z = 0; z < 8; ++z) t[z] = o[e + z] * inv;
                st16(orow + c * 16 + e, t);
              }
            }
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512) : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;
std::once_flag g_once;

bool init_attn() {
  std::call_once(g_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    cudaFuncSetAttribute(k_attn_tc<72>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ACfg<72>::SMEM);
    cudaFuncSetAttribute(k_attn_tc<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ACfg<128>::SMEM);
    cudaFuncSetAttribute(k_attn_tc<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ACfg<64>::SMEM);
  });
  return g_enc != nullptr;
}

template <int D>
cudaError_t attn_tc_t(const AttnArgs& a, cudaStream_t s) {
  // 3-D view of the fused qkv rows: (element within a head, head slot over
  // the q | k | v sections, row); the box is 64 elements x 1 head x 128 rows
  // and elements past the head width read as zero.
  const long long rows = (long long)a.B * (a.Nt + a.Ni);
  CUtensorMap tm;
  cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)(3 * a.H), (cuuint64_t)rows};
  cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)a.ld_qkv * 2};
  cuuint32_t box[3] = {64, 1, 128};
  cuuint32_t estr[3] = {1, 1, 1};
  if (g_enc(&tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.q), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  dim3 grid((a.Nt + 127) / 128 + (a.Ni + 127) / 128, a.H, a.B);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)D);
  k_attn_tc<D><<<grid, ATHREADS, ACfg<D>::SMEM, s>>>(tm, a, scale_log2);
  return launched();
}

}  // namespace

// Tensor-core path when the q/k/v columns of a head can be described by one
// 3-D tensor map over the fused qkv rows: q, k, v sections adjacent (k = q + C,
// v = q + 2C), 16-byte aligned base and row stride.
cudaError_t attention_tc(const AttnArgs& a, cudaStream_t s) {
  if (!init_attn()) return cudaErrorNotSupported;
  const int C = a.H * a.hd;
  const char* q = reinterpret_cast<const char*>(a.q);
  if (reinterpret_cast<const char*>(a.k) != q + 2 * (size_t)C || reinterpret_cast<const char*>(a.v) != q + 4 * (size_t)C)
    return cudaErrorInvalidValue;
  if (((uintptr_t)q & 15) || (a.ld_qkv % 8) || (a.ld_out % 8)) return cudaErrorInvalidValue;
  switch (a.hd) {
    case 64: return attn_tc_t<64>(a, s);
    case 72: return attn_tc_t<72>(a, s);
    case 128: return attn_tc_t<128>(a, s);
    default: return cudaErrorInvalidValue;
  }
}

unsigned int attention_tc_watchdog_take() {
  unsigned int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_attn_watchdog, sizeof(v)) != cudaSuccess) return 0;
  if (v) cudaMemcpyToSymbol(g_attn_watchdog, &z, sizeof(z));
  return v;
}

}  // namespace ff
