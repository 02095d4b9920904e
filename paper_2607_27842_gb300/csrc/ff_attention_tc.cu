// Non-causal attention softmax(q k^T / sqrt(d)) v of the exact block (Eq. 1)
// on the 5th-generation tensor cores, bf16 in, fp32 accumulate.
//
// One CTA per (sample, head, pair of 128-query tiles), 10 warps (sequences
// of at most four key tiles: 6 warps, two CTAs per SM, each CTA taking one
// or more query tiles of its (sample, head) in turn):
//   warp 0     TMA producer: both query tiles once, then key and value tiles
//              of 128 tokens into separate rings, straight from the fused qkv
//              activation (3-D tensor map: head width, head slot, row; the
//              head width is zero-padded to a multiple of 64 by the map);
//   warp 1     TMEM allocator and MMA issuer (the whole warp runs the loop,
//              one elected lane issues).  Per key tile j and query tile i:
//              S_i = Q_i K_j^T into TMEM (both operands K-major from shared
//              memory), then O_i += P_i V_j with P_i read from TMEM (where the
//              softmax wrote it over S_i) and V MN-major from its TMA tile.
//              S_i for tile j + 1 is issued right behind O_i's update for
//              tile j, so one query tile's softmax overlaps the other's MMAs.
//              The issuing thread runs only a few MMAs ahead of the tensor
//              pipe, so every gap between two groups of MMAs holds at most
//              one barrier wait;
//   warps 2-5  softmax of query tile 0, warps 6-9 of query tile 1: each
//              thread owns one query row (its TMEM lane): row max, exp2,
//              row sum, P as bf16 pairs back into TMEM; O is rescaled in TMEM
//              only when the running max grew by more than 2^8 (the final
//              division uses the same stale max, so the result is unchanged).
//              The two warpgroups run freely (making them take turns for
//              the exponentials measured slower once the MMA issue stopped
//              stalling).
// TMEM columns: S_0 [0,128), S_1 [128,256), O_0 [256,384), O_1 [384,512);
// with one query tile per CTA (short sequences): S [0,128), O [128,256).
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

constexpr int AQ = 128;        // queries per tile (MMA M)
constexpr int AKV = 128;       // keys per tile (MMA N of S, K of P V)
constexpr float RESCALE_LOG2 = 8.0f;
constexpr int SHORT_KV_TILES = 4;  // sequences of at most 4 x 128 tokens: one query tile per CTA
constexpr size_t SMEM_LIMIT = 232448;  // opt-in dynamic shared memory per block

__device__ unsigned int g_attn_watchdog;

// Every hand-off in this kernel (S ready -> softmax -> P ready -> MMA) is on
// the critical path, so waits poll instead of suspending.
__device__ __forceinline__ bool wait_a(uint64_t* b, uint32_t parity, volatile int* abort_flag) {
  return mbar_wait<true>(b, parity, abort_flag, &g_attn_watchdog);
}
// the MMA warp's waits: every lane polls, the vote makes the outcome (and so
// the loop control and the operand descriptors behind it) warp-uniform
__device__ __forceinline__ bool wait_u(uint64_t* b, uint32_t parity, volatile int* abort_flag) {
  const bool ok = mbar_test(b, parity) || wait_a(b, parity, abort_flag);
  return __all_sync(0xffffffffu, ok);
}

// QT query tiles per CTA.  QT = 2: two softmax warpgroups that overlap
// each other's MMAs, key / value rings as deep as shared memory allows, one
// CTA per SM.  QT = 1 (short sequences, a couple of key tiles): one softmax
// warpgroup, single-slot rings and half the TMEM, so two CTAs share an SM
// and overlap their latency chains instead; a CTA takes several query tiles
// in turn so that all CTAs fit in one wave and a tile's loads overlap the
// previous tile's tail.
template <int D, int QT> struct ACfg {
  static constexpr int SOFT_WARP0 = 2;                   // first softmax warp
  static constexpr int THREADS = 32 * SOFT_WARP0 + 128 * QT;  // TMA warp, MMA warp, softmax warpgroups
  static constexpr int NBOX = D <= 64 ? 1 : 2;           // 64-wide column boxes per tile row
  static constexpr int DK = (D + 15) / 16 * 16;          // q k^T reduction width and P V output width
  static constexpr uint32_t BOX = 128 * 128;             // one [128 rows x 64] bf16 box, 16 KB
  static constexpr uint32_t TILE = NBOX * BOX;           // one Q, K or V tile
  static constexpr int NST = (int)((SMEM_LIMIT - 1024 - 512 - QT * (size_t)TILE) / TILE);
  static constexpr int KST = QT == 1 ? 1 : NST >= 8 ? 4 : (NST + 1) / 2;  // key ring depth
  static constexpr int VST = QT == 1 ? 1 : NST >= 8 ? 4 : NST / 2;        // value ring depth
  static constexpr size_t SMEM = 1024 + (size_t)(QT + KST + VST) * TILE + 512;
  static constexpr uint32_t TMEM_O = QT * AKV;           // S_i at i * 128, O_i at TMEM_O + i * 128
  static constexpr uint32_t TMEM_COLS = QT == 1 ? 256 : 512;
  // kind::f16, D fp32, A/B bf16; S: both K-major, N = 128; O: A (P) from
  // TMEM, B (V) MN-major (bit 16), N = DK
  static constexpr uint32_t IDESC_S = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(AKV >> 3) << 17) |
                                      ((uint32_t)(AQ >> 4) << 24);
  static constexpr uint32_t IDESC_O = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) | ((uint32_t)(DK >> 3) << 17) |
                                      ((uint32_t)(AQ >> 4) << 24);
  static_assert(KST >= 1 && VST >= 1 && (QT == 1 || KST >= 2), "shared memory too small for the key/value rings");
  static_assert(SMEM <= SMEM_LIMIT, "shared memory budget");
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

// D[tmem] (+)= A[tmem] * B[smem]: A is read from TMEM (row m = lane m, two
// bf16 per 32-bit column along K)
__device__ __forceinline__ void umma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t accum) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(
          d_tmem),
      "r"(a_tmem), "l"(b), "r"(idesc), "r"(accum));
}

// 64 consecutive 32-bit TMEM columns of this warp's 32 lanes, waited for in
// the same statement so no use of the registers can precede the wait
__device__ __forceinline__ void tmem_ld64w(uint32_t taddr, float* v) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63}, [%64];\n"
      "tcgen05.wait::ld.sync.aligned;\n"
      : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]), "=f"(v[4]), "=f"(v[5]), "=f"(v[6]), "=f"(v[7]), "=f"(v[8]), "=f"(v[9]), "=f"(v[10]), "=f"(v[11]), "=f"(v[12]), "=f"(v[13]), "=f"(v[14]), "=f"(v[15]), "=f"(v[16]), "=f"(v[17]), "=f"(v[18]), "=f"(v[19]), "=f"(v[20]), "=f"(v[21]), "=f"(v[22]), "=f"(v[23]), "=f"(v[24]), "=f"(v[25]), "=f"(v[26]), "=f"(v[27]), "=f"(v[28]), "=f"(v[29]), "=f"(v[30]), "=f"(v[31]), "=f"(v[32]), "=f"(v[33]), "=f"(v[34]), "=f"(v[35]), "=f"(v[36]), "=f"(v[37]), "=f"(v[38]), "=f"(v[39]), "=f"(v[40]), "=f"(v[41]), "=f"(v[42]), "=f"(v[43]), "=f"(v[44]), "=f"(v[45]), "=f"(v[46]), "=f"(v[47]), "=f"(v[48]), "=f"(v[49]), "=f"(v[50]), "=f"(v[51]), "=f"(v[52]), "=f"(v[53]), "=f"(v[54]), "=f"(v[55]), "=f"(v[56]), "=f"(v[57]), "=f"(v[58]), "=f"(v[59]), "=f"(v[60]), "=f"(v[61]), "=f"(v[62]), "=f"(v[63])
      : "r"(taddr)
      : "memory");
}
// 32 TMEM columns without waiting; tmem_wait32 on the same registers
// completes them (its in/out operands keep every use behind the wait)
__device__ __forceinline__ void tmem_ld32_async(uint32_t taddr, float* v) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n"
               : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]), "=f"(v[4]), "=f"(v[5]), "=f"(v[6]), "=f"(v[7]), "=f"(v[8]), "=f"(v[9]), "=f"(v[10]), "=f"(v[11]), "=f"(v[12]), "=f"(v[13]), "=f"(v[14]), "=f"(v[15]), "=f"(v[16]), "=f"(v[17]), "=f"(v[18]), "=f"(v[19]), "=f"(v[20]), "=f"(v[21]), "=f"(v[22]), "=f"(v[23]), "=f"(v[24]), "=f"(v[25]), "=f"(v[26]), "=f"(v[27]), "=f"(v[28]), "=f"(v[29]), "=f"(v[30]), "=f"(v[31])
               : "r"(taddr)
               : "memory");
}
__device__ __forceinline__ void tmem_wait32(float* v) {
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" : "+f"(v[0]), "+f"(v[1]), "+f"(v[2]), "+f"(v[3]), "+f"(v[4]), "+f"(v[5]), "+f"(v[6]), "+f"(v[7]), "+f"(v[8]), "+f"(v[9]), "+f"(v[10]), "+f"(v[11]), "+f"(v[12]), "+f"(v[13]), "+f"(v[14]), "+f"(v[15]), "+f"(v[16]), "+f"(v[17]), "+f"(v[18]), "+f"(v[19]), "+f"(v[20]), "+f"(v[21]), "+f"(v[22]), "+f"(v[23]), "+f"(v[24]), "+f"(v[25]), "+f"(v[26]), "+f"(v[27]), "+f"(v[28]), "+f"(v[29]), "+f"(v[30]), "+f"(v[31]) : : "memory");
}
__device__ __forceinline__ void tmem_st16u(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};\n" ::"r"(taddr),
               "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
               "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
               : "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};\n" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
        "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]),
        "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// packed pairs of fp32 (one 64-bit register pair): a.x + 2^32 * a.y
__device__ __forceinline__ unsigned long long f2u(float a, float b) {
  return (unsigned long long)__float_as_uint(a) | ((unsigned long long)__float_as_uint(b) << 32);
}
__device__ __forceinline__ unsigned long long ffma2(unsigned long long a, unsigned long long b, unsigned long long c) {
  unsigned long long r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
__device__ __forceinline__ unsigned long long fadd2(unsigned long long a, unsigned long long b) {
  unsigned long long r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ float lo_f(unsigned long long x) { return __uint_as_float((unsigned)x); }
__device__ __forceinline__ float hi_f(unsigned long long x) { return __uint_as_float((unsigned)(x >> 32)); }

// 16 pairs of S (v[2e], v[2e + 1]) -> exp2(s * scale - m) as bf16 pairs,
// their sum added to the packed accumulators
__device__ __forceinline__ void exp_pairs16(const float* v, unsigned long long sc2, unsigned long long nm2,
                                            unsigned long long (&acc2)[4], uint32_t (&pk)[16]) {
#pragma unroll
  for (int e = 0; e < 16; ++e) {
    const unsigned long long x = ffma2(f2u(v[2 * e], v[2 * e + 1]), sc2, nm2);
    const float p0 = ex2(lo_f(x)), p1 = ex2(hi_f(x));
    acc2[e & 3] = fadd2(acc2[e & 3], f2u(p0, p1));
    __nv_bfloat162 t2 = __floats2bfloat162_rn(p0, p1);
    pk[e] = *reinterpret_cast<uint32_t*>(&t2);
  }
}
__device__ __forceinline__ float acc_total(const unsigned long long (&acc2)[4]) {
  const unsigned long long a = fadd2(fadd2(acc2[0], acc2[1]), fadd2(acc2[2], acc2[3]));
  return lo_f(a) + hi_f(a);
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
// number of valid rows (<= 0 for a tile past the sequence end).
struct SegTile {
  int row0, valid;
};
__device__ __forceinline__ SegTile seg_tile(const AttnArgs& a, int b, int t) {
  const int nt_tiles = (a.Nt + 127) / 128;
  if (t < nt_tiles) return {b * a.Nt + t * 128, min(128, a.Nt - t * 128)};
  const int u = t - nt_tiles;
  return {a.B * a.Nt + b * a.Ni + u * 128, min(128, a.Ni - u * 128)};
}

template <int D, int QT>
__global__ void __launch_bounds__(ACfg<D, QT>::THREADS, QT == 1 ? 2 : 1)
    k_attn_tc(const __grid_constant__ CUtensorMap tmQKV, AttnArgs a, float scale_log2, int ipc) {
  using C = ACfg<D, QT>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;                        // QT tiles
  uint8_t* sK = sQ + QT * C::TILE;           // KST tiles
  uint8_t* sV = sK + C::KST * C::TILE;       // VST tiles
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + C::VST * C::TILE);
  uint64_t* q_full = bars;
  uint64_t* k_full = q_full + 1;
  uint64_t* k_empty = k_full + C::KST;
  uint64_t* v_full = k_empty + C::KST;
  uint64_t* v_empty = v_full + C::VST;
  uint64_t* s_full = v_empty + C::VST;       // per query tile
  uint64_t* p_ready = s_full + 2;            // per query tile
  uint64_t* o_final = p_ready + 2;
  uint64_t* q_empty = o_final + 1;           // Q tiles free for the CTA's next item
  uint64_t* o_free = q_empty + 1;            // O read out by the softmax warps' epilogue
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(o_free + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y, b = blockIdx.z;
  const int nkv = (a.Nt + 127) / 128 + (a.Ni + 127) / 128;  // key tiles = query tiles of a sample
  // item it of this CTA: query tiles QT * (blockIdx.x * ipc + it) + i; the
  // key / value rings, s_full and p_ready count on across items (kv step
  // jj = it * nkv + j)
  auto item_live = [&](int it) { return QT * (blockIdx.x * ipc + it) < nkv; };

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < C::KST; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < C::VST; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int i = 0; i < QT; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_ready[i], 128);
    }
    mbar_init(o_final, 1);
    mbar_init(q_empty, 1);
    mbar_init(o_free, 128 * QT);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmQKV) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(tmem_slot)),
                 "r"(C::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // dependents may launch once every CTA holds its TMEM; the previous
  // kernel's outputs are complete after the wait
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      int nk = 0, nv = 0, q_last = -1;
      bool ok = true;
      for (int it = 0; it < ipc && ok && item_live(it); ++it) {
        // the next item's Q waits for the previous item's last S MMAs
        if (it > 0 && !wait_a(q_empty, (it - 1) & 1, abort_flag)) break;
        mbar_expect_tx(q_full, QT * C::TILE);
        for (int i = 0; i < QT; ++i) {
          const SegTile qs = seg_tile(a, b, QT * (blockIdx.x * ipc + it) + i);
          for (int bx = 0; bx < C::NBOX; ++bx)
            tma_load3(&tmQKV, q_full, sQ + i * C::TILE + bx * C::BOX, 64 * bx, h, qs.row0);
        }
        q_last = it;
        for (int j = 0; j < nkv; ++j) {
          const int jj = it * nkv + j;
          const SegTile ks = seg_tile(a, b, j);
          const int sk = jj % C::KST, sv = jj % C::VST;
          if (!wait_a(&k_empty[sk], ((jj / C::KST) & 1) ^ 1, abort_flag)) { ok = false; break; }
          mbar_expect_tx(&k_full[sk], C::TILE);
          for (int bx = 0; bx < C::NBOX; ++bx)
            tma_load3(&tmQKV, &k_full[sk], sK + sk * C::TILE + bx * C::BOX, 64 * bx, a.H + h, ks.row0);
          ++nk;
          if (!wait_a(&v_empty[sv], ((jj / C::VST) & 1) ^ 1, abort_flag)) { ok = false; break; }
          mbar_expect_tx(&v_full[sv], C::TILE);
          for (int bx = 0; bx < C::NBOX; ++bx)
            tma_load3(&tmQKV, &v_full[sv], sV + sv * C::TILE + bx * C::BOX, 64 * bx, 2 * a.H + h, ks.row0);
          ++nv;
        }
      }
      // Copies still in flight complete on their full barriers; wait for the
      // last ring's worth of each so none lands after the CTA exits.
      for (int k = 0; k < C::KST && k < nk; ++k) {
        const int j = nk - 1 - k;
        const unsigned long long t0 = gtimer();
        while (!mbar_try(&k_full[j % C::KST], (j / C::KST) & 1))
          if (gtimer() - t0 > WAIT_LIMIT_NS) { atomicOr(&g_attn_watchdog, 2u); break; }
      }
      for (int k = 0; k < C::VST && k < nv; ++k) {
        const int j = nv - 1 - k;
        const unsigned long long t0 = gtimer();
        while (!mbar_try(&v_full[j % C::VST], (j / C::VST) & 1))
          if (gtimer() - t0 > WAIT_LIMIT_NS) { atomicOr(&g_attn_watchdog, 2u); break; }
      }
      // and the last item's query tiles (phase q_last of q_full; on the
      // normal path the MMA warp has already seen it complete)
      if (q_last >= 0) {
        const unsigned long long t0 = gtimer();
        while (!mbar_try(q_full, q_last & 1))
          if (gtimer() - t0 > WAIT_LIMIT_NS) { atomicOr(&g_attn_watchdog, 2u); break; }
      }
    }
  } else if (warp == 1) {
    bool ok = true;
    const uint64_t qd0 = sw128_desc(saddr(sQ)), qd1 = sw128_desc(saddr(sQ + C::TILE));
    // S_i = Q_i K_jj^T (DK / 16 steps of 16 along the head width: box k / 4,
    // +32 B per step inside the box), then arrive on s_full[i]
    auto issue_s = [&](int i, int jj) {
      const uint64_t kd = sw128_desc(saddr(sK + (jj % C::KST) * C::TILE));
      const uint64_t qd = i ? qd1 : qd0;
#pragma unroll
      for (int k = 0; k < C::DK / 16; ++k) {
        const uint64_t off = (uint64_t)((k >> 2) * (C::BOX >> 4) + 2 * (k & 3));
        if (elect_one()) umma(tmem + (uint32_t)(i * AKV), qd + off, kd + off, C::IDESC_S, k != 0);
      }
      if (elect_one()) umma_commit(&s_full[i]);
    };
    for (int it = 0; it < ipc && ok && item_live(it); ++it) {
      const int jb = it * nkv;  // the item's first kv step
      ok = wait_u(q_full, it & 1, abort_flag);
      if (ok) ok = wait_u(&k_full[jb % C::KST], (jb / C::KST) & 1, abort_flag);
      if (!ok) break;
      tc_fence_after();
      issue_s(0, jb);
      if (QT == 2) issue_s(1, jb);
      if (elect_one()) umma_commit(&k_empty[jb % C::KST]);
      if (nkv == 1 && elect_one()) umma_commit(q_empty);  // the item's last S MMAs
      ok = wait_u(&v_full[jb % C::VST], (jb / C::VST) & 1, abort_flag);
      // the previous item's O has been read out before this item's first P V
      if (ok && it > 0) ok = wait_u(o_free, (it - 1) & 1, abort_flag);
      // Per key tile j: [p_ready 0] O_0 += P_0 V_j [k_full j+1] S_0 for j + 1
      // [p_ready 1] O_1 += P_1 V_j [v_full j+1] S_1 for j + 1 -- one wait in
      // each gap between MMA groups
      for (int j = 0; j < nkv && ok; ++j) {
        const int jj = jb + j;
        const int sv = jj % C::VST;
        const bool more = j + 1 < nkv;
        const uint32_t vaddr = saddr(sV + sv * C::TILE);
        for (int i = 0; i < QT; ++i) {
          ok = wait_u(&p_ready[i], jj & 1, abort_flag);
          if (!ok) break;
          tc_fence_after();
          // O_i += P_i V_j: 16 keys per step = 8 TMEM columns of P, 2 groups
          // of 8 value rows (2 KB) of the MN-major V tile
#pragma unroll
          for (int k = 0; k < AKV / 16; ++k) {
            const uint64_t vd = sw128_desc_mn(vaddr + (uint32_t)k * 2048u, C::BOX);
            if (elect_one())
              umma_ts(tmem + C::TMEM_O + (uint32_t)(i * AKV), tmem + (uint32_t)(i * AKV + k * 8), vd, C::IDESC_O,
                      (j | k) != 0);
          }
          if (i == QT - 1 && elect_one()) umma_commit(&v_empty[sv]);
          if (more) {
            if (i == 0) ok = wait_u(&k_full[(jj + 1) % C::KST], ((jj + 1) / C::KST) & 1, abort_flag);
            if (ok && i == QT - 1) ok = wait_u(&v_full[(jj + 1) % C::VST], ((jj + 1) / C::VST) & 1, abort_flag);
            if (!ok) break;
            tc_fence_after();
            issue_s(i, jj + 1);  // behind O_i's update: the MMA pipe reads P_i before S_i is overwritten
            if (i == QT - 1 && elect_one()) {
              umma_commit(&k_empty[(jj + 1) % C::KST]);
              if (j + 2 == nkv) umma_commit(q_empty);  // the item's last S MMAs
            }
          }
        }
      }
      if (ok && elect_one()) umma_commit(o_final);
    }
  } else if (warp >= C::SOFT_WARP0) {
    // softmax of query tile i: row r of the tile = TMEM lane r
    const int i = (warp - C::SOFT_WARP0) >> 2;
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const uint32_t s_col = tmem + lane_off + (uint32_t)(i * AKV);
    const uint32_t o_col = tmem + lane_off + C::TMEM_O + (uint32_t)(i * AKV);
    bool ok = true;
    for (int it = 0; it < ipc && ok && item_live(it); ++it) {
    const SegTile qs = seg_tile(a, b, QT * (blockIdx.x * ipc + it) + i);
    float m = -INFINITY, l = 0.f;
    for (int j = 0; j < nkv; ++j) {
      const int valid = seg_tile(a, b, j).valid;
      int w = 1;
      if (lane == 0) w = wait_a(&s_full[i], (it * nkv + j) & 1, abort_flag) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
      tc_fence_after();
      // row max as a tree of three-input maxima (72 instructions for 128
      // values instead of 127).  One query tile per CTA (short sequences,
      // latency-bound): S is read 64 columns at a time for the max and again
      // in quarters for the exponentials, which keeps the row out of
      // registers; two query tiles: the row is held in registers.
      float v[QT == 1 ? 1 : AKV];
      float mx[16];
      if constexpr (QT == 2) {
        // Speculative softmax: exponentials against the running reference
        // m while S streams in from TMEM, P stored as it is made.  They are
        // the lazy-rescale result whenever no exponent exceeds 2^8, which a
        // tile sum <= 256 guarantees; otherwise (and on the first tile) the
        // row max is taken from the registers, O is rescaled if the max
        // grew by more than 2^8, and P is recomputed.
        const unsigned long long sc2 = f2u(scale_log2, scale_log2);
        bool need = true;
        float lt = 0.f;
        if (j > 0) {
          const unsigned long long nm2 = f2u(-m, -m);
          unsigned long long acc2[4] = {0ull, 0ull, 0ull, 0ull};
          tmem_ld32_async(s_col, v);
          tmem_wait32(v);
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            // S columns [32 (k + 1), 32 (k + 2)) load while chunk k is
            // finished; P chunk k goes to columns [16 k, 16 k + 16), which
            // hold S already read
            if (k + 1 < 4) tmem_ld32_async(s_col + (uint32_t)(32 * (k + 1)), v + 32 * (k + 1));
            if (valid < AKV) {
#pragma unroll
              for (int e = 0; e < 32; ++e)
                if (32 * k + e >= valid) v[32 * k + e] = -INFINITY;
            }
            uint32_t pk[16];
            exp_pairs16(v + 32 * k, sc2, nm2, acc2, pk);
            tmem_st16u(s_col + (uint32_t)(16 * k), pk);
            if (k + 1 < 4) tmem_wait32(v + 32 * (k + 1));
          }
          lt = acc_total(acc2);
          need = __any_sync(0xffffffffu, !(lt <= 256.0f));   // also a non-finite sum
        } else {
          tmem_ld64w(s_col, v);
          tmem_ld64w(s_col + 64, v + 64);
          if (valid < AKV) {
#pragma unroll
            for (int e = 0; e < AKV; ++e)
              if (e >= valid) v[e] = -INFINITY;
          }
        }
        float alpha = 1.0f;
        if (need) {
#pragma unroll
          for (int e = 0; e < 16; ++e)
            mx[e] = max3f(max3f(v[e], v[e + 16], v[e + 32]), max3f(v[e + 48], v[e + 64], v[e + 80]),
                          fmaxf(v[e + 96], v[e + 112]));
#pragma unroll
          for (int e = 0; e < 5; ++e) mx[e] = max3f(mx[e], mx[e + 5], mx[e + 10]);
          mx[0] = max3f(max3f(mx[0], mx[1], mx[2]), max3f(mx[3], mx[4], mx[15]), mx[0]);
          const float m_new = fmaxf(m, mx[0] * scale_log2);
          const bool grow = m_new > m + RESCALE_LOG2;  // always on the first tile
          if (__any_sync(0xffffffffu, grow)) {
            alpha = grow ? ex2(m - m_new) : 1.0f;
            // O_i holds every update through tile j - 1: s_full[i] for tile
            // j arrived after them
            if (j >= 1) {
#pragma unroll
              for (int c = 0; c < C::DK / 16; ++c) {
                float o[16];
                tmem_ld16(o_col + (uint32_t)(c * 16), o);
#pragma unroll
                for (int e = 0; e < 16; ++e) o[e] *= alpha;
                tmem_st16(o_col + (uint32_t)(c * 16), o);
              }
            }
            if (grow) m = m_new;
            tmem_st_wait();   // the speculative P stores land before their recomputation
            const unsigned long long nm2 = f2u(-m, -m);
            unsigned long long acc2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              uint32_t pk[16];
              exp_pairs16(v + 32 * k, sc2, nm2, acc2, pk);
              tmem_st16u(s_col + (uint32_t)(16 * k), pk);
            }
            lt = acc_total(acc2);
          }
        }
        l = l * alpha + lt;
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&p_ready[i]);
        continue;
      }
      if constexpr (QT == 1) {
#pragma unroll
        for (int e = 0; e < 16; ++e) mx[e] = -INFINITY;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          float t[64];
          tmem_ld64w(s_col + (uint32_t)(64 * hh), t);
          if (valid < AKV) {
#pragma unroll
            for (int e = 0; e < 64; ++e)
              if (64 * hh + e >= valid) t[e] = -INFINITY;
          }
#pragma unroll
          for (int e = 0; e < 16; ++e) mx[e] = max3f(mx[e], max3f(t[e], t[e + 16], t[e + 32]), t[e + 48]);
        }
      } else {
        tmem_ld64w(s_col, v);
        tmem_ld64w(s_col + 64, v + 64);
        if (valid < AKV) {
#pragma unroll
          for (int e = 0; e < AKV; ++e)
            if (e >= valid) v[e] = -INFINITY;
        }
#pragma unroll
        for (int e = 0; e < 16; ++e)
          mx[e] = max3f(max3f(v[e], v[e + 16], v[e + 32]), max3f(v[e + 48], v[e + 64], v[e + 80]),
                        fmaxf(v[e + 96], v[e + 112]));
      }
#pragma unroll
      for (int e = 0; e < 5; ++e) mx[e] = max3f(mx[e], mx[e + 5], mx[e + 10]);
      mx[0] = max3f(max3f(mx[0], mx[1], mx[2]), max3f(mx[3], mx[4], mx[15]), mx[0]);
      const float m_new = fmaxf(m, mx[0] * scale_log2);
      const bool grow = m_new > m + RESCALE_LOG2;  // also true on the first tile
      const float m_use = grow ? m_new : m;
      const float alpha = grow ? ex2(m - m_new) : 1.0f;
      // O_i holds every update through tile j - 1: s_full[i] for tile j
      // arrived after them
      if (j >= 1 && __any_sync(0xffffffffu, grow)) {
#pragma unroll
        for (int c = 0; c < C::DK / 16; ++c) {
          float o[16];
          tmem_ld16(o_col + (uint32_t)(c * 16), o);
#pragma unroll
          for (int e = 0; e < 16; ++e) o[e] *= alpha;
          tmem_st16(o_col + (uint32_t)(c * 16), o);
        }
      }
      m = m_use;
      float ls[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) ls[e] = 0.f;
      // P as bf16 pairs into the first 64 columns of S_i (already read)
      if constexpr (QT == 1) {
        // S again, 32 columns at a time (the next quarter loading while this
        // one is finished); quarter k's P columns [16k, 16k + 16) lie in
        // columns already read
        float sq[2][32];
        tmem_ld32_async(s_col, sq[0]);
        tmem_wait32(sq[0]);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if (k + 1 < 4) tmem_ld32_async(s_col + (uint32_t)(32 * (k + 1)), sq[(k + 1) & 1]);
          float* x = sq[k & 1];
          if (valid < AKV) {
#pragma unroll
            for (int e = 0; e < 32; ++e)
              if (32 * k + e >= valid) x[e] = -INFINITY;
          }
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const float p0 = ex2(fmaf(x[2 * e], scale_log2, -m));
            const float p1 = ex2(fmaf(x[2 * e + 1], scale_log2, -m));
            ls[e & 7] += p0 + p1;
            __nv_bfloat162 t2 = __floats2bfloat162_rn(p0, p1);
            pk[e] = *reinterpret_cast<uint32_t*>(&t2);
          }
          tmem_st16u(s_col + (uint32_t)(16 * k), pk);
          if (k + 1 < 4) tmem_wait32(sq[(k + 1) & 1]);
        }
      } else {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          uint32_t pk[32];
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float p0 = ex2(fmaf(v[half * 64 + 2 * e], scale_log2, -m));
            const float p1 = ex2(fmaf(v[half * 64 + 2 * e + 1], scale_log2, -m));
            ls[e & 7] += p0 + p1;
            __nv_bfloat162 t2 = __floats2bfloat162_rn(p0, p1);
            pk[e] = *reinterpret_cast<uint32_t*>(&t2);
          }
          tmem_st32(s_col + (uint32_t)(half * 32), pk);
        }
      }
      l = l * alpha + (((ls[0] + ls[1]) + (ls[2] + ls[3])) + ((ls[4] + ls[5]) + (ls[6] + ls[7])));
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&p_ready[i]);
    }
    if (!ok) break;
    int w = 1;
    if (lane == 0) w = wait_a(o_final, it & 1, abort_flag) ? 1 : 0;
    if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
    tc_fence_after();
    const float inv = 1.0f / l;
    bf16* orow = reinterpret_cast<bf16*>(a.out) + (size_t)(qs.row0 + (r < qs.valid ? r : 0)) * a.ld_out + (size_t)h * D;
#pragma unroll
    for (int c = 0; c < C::DK / 16; ++c) {
      float o[16];
      tmem_ld16(o_col + (uint32_t)(c * 16), o);
      if (r < qs.valid) {
#pragma unroll
        for (int e = 0; e < 16; e += 8) {
          if (c * 16 + e < D) {
            float t8[8];
#pragma unroll
            for (int z = 0; z < 8; ++z) t8[z] = o[e + z] * inv;
            st16(orow + c * 16 + e, t8);
          }
        }
      }
    }
    // O is read out: the next item's first P V may overwrite it
    tc_fence_before();
    mbar_arrive(o_free);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::TMEM_COLS) : "memory");
  }
}


// ---------------------------------------------------------------------------
// Sequences of at most two key tiles (256 tokens; DiT-XL/2) with a head
// width of at most 80: one query tile at a time, two CTAs per SM, every CTA
// taking the query tiles of one (sample, head) in turn.  The head's K and V
// tiles are loaded once and stay resident for all of the CTA's query tiles;
// S over all keys comes from one N = 256 MMA, so the softmax needs no online
// rescaling (one pass for the row max, one for P).  Head widths over 64 keep
// their last 16 columns in separate 32-byte-swizzled boxes (4 KB per tile
// instead of a second 16 KB box), which lets Q, both K and both V tiles of a
// 72-wide head fit two CTAs per SM.  TMEM (256 columns): S in [0, 256), P
// over its first half, O in [128, 128 + DK) once the softmax has read S.
// ---------------------------------------------------------------------------
template <int D> struct ACfgShort {
  static constexpr int DK = (D + 15) / 16 * 16;      // 64 or 80
  static constexpr bool TAIL = DK > 64;
  static constexpr uint32_t MAIN = 128 * 128;        // [128 rows x 64] bf16, 128-byte swizzle
  static constexpr uint32_t TAILB = 128 * 32;        // [128 rows x 16] bf16, 32-byte swizzle
  static constexpr uint32_t BYTES_Q = MAIN + (TAIL ? TAILB : 0);   // one tile of q, k or v
  static constexpr int THREADS = 192;
  static constexpr uint32_t TMEM_COLS = 256;
  // kind::f16, D fp32, A/B bf16; S: both K-major, N set per launch (128 or
  // 256); O: A (P) from TMEM, B (V) MN-major, N = 64 (+ 16 for the tail)
  static constexpr uint32_t IDESC_S128 = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(128 >> 3) << 17) |
                                         ((uint32_t)(AQ >> 4) << 24);
  static constexpr uint32_t IDESC_S256 = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(256 >> 3) << 17) |
                                         ((uint32_t)(AQ >> 4) << 24);
  static constexpr int VN = (DK + 31) / 32 * 32;     // P V width: whole 32-column boxes (64 or 96)
  static constexpr uint32_t IDESC_O = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) | ((uint32_t)(VN >> 3) << 17) |
                                      ((uint32_t)(AQ >> 4) << 24);
  static constexpr uint32_t VBOX = 128 * 64;          // [128 keys x 32] bf16, 64-byte swizzle
  static constexpr uint32_t VTILE = (VN / 32) * VBOX; // a V tile: VN / 32 such boxes along the head width
};
// shared-memory layout of the short kernel (offsets from the 1 KB-aligned base)
struct ShortLayout {
  static constexpr uint32_t QA = 0;          // 16 KB
  static constexpr uint32_t QT = 16384;      // 4 KB
  static constexpr uint32_t KA = 20480;      // 2 x 16 KB, adjacent: one 256-row K-major operand
  static constexpr uint32_t KT = 53248;      // 2 x 4 KB, adjacent
  static constexpr uint32_t VA = 61440;      // 2 x 24 KB: tile j, head columns 32i .. 32i + 31 at + 24 KB j + 8 KB i
  static constexpr uint32_t BARS = 110592;   // barriers, TMEM slot, abort flag
  static constexpr size_t SMEM = 1024 + 110592 + 256;   // two CTAs per SM
};
static_assert(ShortLayout::KA % 1024 == 0 && ShortLayout::VA % 1024 == 0 && ShortLayout::QT % 1024 == 0 &&
                  ShortLayout::KT % 1024 == 0 && ShortLayout::VA + 2 * 3 * 8192 <= ShortLayout::BARS,
              "swizzle atoms need 1 KB-aligned tiles");

// K-major operand with 32-byte swizzle: 8-row groups 256 B apart
__device__ __forceinline__ uint64_t sw32_desc(uint32_t addr) {
  uint64_t d = (uint64_t)((addr & 0x3FFFF) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(256 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)6 << 61;
  return d;
}
// MN-major operand with 64-byte swizzle: 32-element atoms along N 8 KB
// apart (one [128 x 32] box each), 8 rows along K per 512-byte group
__device__ __forceinline__ uint64_t sw64_desc_mn(uint32_t addr) {
  uint64_t d = (uint64_t)((addr & 0x3FFFF) >> 4);
  d |= (uint64_t)(8192 >> 4) << 16;
  d |= (uint64_t)(512 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)4 << 61;
  return d;
}

template <int D>
__global__ void __launch_bounds__(192, 2)
    k_attn_short(const __grid_constant__ CUtensorMap tmQKV, const __grid_constant__ CUtensorMap tmTail,
                 const __grid_constant__ CUtensorMap tmV, AttnArgs a, float scale_log2, int ipc) {
  using C = ACfgShort<D>;
  using L = ShortLayout;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BARS);
  uint64_t* q_full = bars;
  uint64_t* k_full = bars + 1;
  uint64_t* v_full = bars + 2;
  uint64_t* s_full = bars + 3;
  uint64_t* p_ready = bars + 4;
  uint64_t* o_final = bars + 5;
  uint64_t* q_empty = bars + 6;
  uint64_t* o_free = bars + 7;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 8);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y, b = blockIdx.z;
  const int nkv = (a.Nt + 127) / 128 + (a.Ni + 127) / 128;   // 1 or 2
  auto item_live = [&](int it) { return blockIdx.x * ipc + it < nkv; };

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(k_full, 1);
    mbar_init(v_full, 1);
    mbar_init(s_full, 1);
    mbar_init(p_ready, 128);
    mbar_init(o_final, 1);
    mbar_init(q_empty, 1);
    mbar_init(o_free, 128);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmQKV) : "memory");
    if (C::TAIL) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmTail) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmV) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(tmem_slot)),
                 "r"(C::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      // a tile of the q (section 0), k (1) or v (2) columns of head h: its
      // 128-byte box and, for head widths over 64, the 32-byte tail box
      bool k_issued = false, v_issued = false;
      int q_last = -1;
      if (item_live(0)) {
        mbar_expect_tx(k_full, (uint32_t)nkv * C::BYTES_Q);
        for (int j = 0; j < nkv; ++j) {
          const int row0 = seg_tile(a, b, j).row0;
          tma_load3(&tmQKV, k_full, smem + L::KA + j * C::MAIN, 0, a.H + h, row0);
          if (C::TAIL) tma_load3(&tmTail, k_full, smem + L::KT + j * C::TAILB, 64, a.H + h, row0);
        }
        k_issued = true;
        for (int it = 0; it < ipc && item_live(it); ++it) {
          if (it > 0 && !wait_a(q_empty, (it - 1) & 1, abort_flag)) break;
          mbar_expect_tx(q_full, C::BYTES_Q);
          const int qrow0 = seg_tile(a, b, blockIdx.x * ipc + it).row0;
          tma_load3(&tmQKV, q_full, smem + L::QA, 0, h, qrow0);
          if (C::TAIL) tma_load3(&tmTail, q_full, smem + L::QT, 64, h, qrow0);
          q_last = it;
          if (it == 0) {
            mbar_expect_tx(v_full, (uint32_t)nkv * C::VTILE);
            for (int j = 0; j < nkv; ++j) {
              const int row0 = seg_tile(a, b, j).row0;
#pragma unroll
              for (int i = 0; i < C::VN / 32; ++i)
                tma_load3(&tmV, v_full, smem + L::VA + j * C::VTILE + i * C::VBOX, 32 * i, 2 * a.H + h, row0);
            }
            v_issued = true;
          }
        }
      }
      // copies still in flight land before the CTA exits
      auto drain = [&](uint64_t* bar, uint32_t parity) {
        const unsigned long long t0 = gtimer();
        while (!mbar_try(bar, parity))
          if (gtimer() - t0 > WAIT_LIMIT_NS) { atomicOr(&g_attn_watchdog, 2u); break; }
      };
      if (k_issued) drain(k_full, 0);
      if (v_issued) drain(v_full, 0);
      if (q_last >= 0) drain(q_full, q_last & 1);
    }
  } else if (warp == 1) {
    bool ok = true;
    const uint32_t base = saddr(smem);
    const uint32_t idesc_s = nkv > 1 ? C::IDESC_S256 : C::IDESC_S128;
    for (int it = 0; it < ipc && ok && item_live(it); ++it) {
      ok = wait_u(q_full, it & 1, abort_flag);
      if (ok && it == 0) ok = wait_u(k_full, 0, abort_flag);
      // O of the previous item is read out before S overwrites its columns
      if (ok && it > 0) ok = wait_u(o_free, (it - 1) & 1, abort_flag);
      if (!ok) break;
      tc_fence_after();
      // S = Q K^T over all keys: 4 steps of 16 in the 128-byte boxes (+32 B
      // per step inside the swizzle atom), then the 32-byte tail box
#pragma unroll
      for (int k = 0; k < C::DK / 16; ++k) {
        const uint64_t ad = k < 4 ? sw128_desc(base + L::QA) + (uint64_t)(2 * k) : sw32_desc(base + L::QT);
        const uint64_t bd = k < 4 ? sw128_desc(base + L::KA) + (uint64_t)(2 * k) : sw32_desc(base + L::KT);
        if (elect_one()) umma(tmem, ad, bd, idesc_s, k != 0);
      }
      if (elect_one()) {
        umma_commit(s_full);
        umma_commit(q_empty);
      }
      ok = wait_u(p_ready, it & 1, abort_flag);
      if (ok && it == 0) ok = wait_u(v_full, 0, abort_flag);
      if (!ok) break;
      tc_fence_after();
      // O = P V: keys 16k .. 16k + 15 are P columns 8k .. 8k + 7; 16 rows of
      // key tile k / 8 (1 KB into each of its 64-byte-swizzled boxes)
      for (int k = 0; k < 8 * nkv; ++k) {
        const int j = k >> 3, kk = k & 7;
        const uint64_t vd = sw64_desc_mn(base + L::VA + j * C::VTILE + (uint32_t)kk * 1024u);
        if (elect_one()) umma_ts(tmem + 128, tmem + (uint32_t)(8 * k), vd, C::IDESC_O, k != 0);
      }
      if (elect_one()) umma_commit(o_final);
    }
  } else {
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const uint32_t s_col = tmem + ((uint32_t)(q * 32) << 16);
    const uint32_t o_col = s_col + 128;
    const int valid0 = seg_tile(a, b, 0).valid;
    const int valid1 = nkv > 1 ? seg_tile(a, b, 1).valid : 0;
    bool ok = true;
    for (int it = 0; it < ipc && ok && item_live(it); ++it) {
      const SegTile qs = seg_tile(a, b, blockIdx.x * ipc + it);
      int w = 1;
      if (lane == 0) w = wait_a(s_full, it & 1, abort_flag) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
      tc_fence_after();
      // pass 1: row max over the keys, 64 columns at a time
      float mx[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) mx[e] = -INFINITY;
#pragma unroll
      for (int c4 = 0; c4 < 4; ++c4) {
        if (c4 >= 2 * nkv) break;
        float t[64];
        tmem_ld64w(s_col + (uint32_t)(64 * c4), t);
        const int vt = (c4 < 2 ? valid0 : valid1) - 64 * (c4 & 1);   // valid keys in these 64 columns
        if (vt < 64) {
#pragma unroll
          for (int e = 0; e < 64; ++e)
            if (e >= vt) t[e] = -INFINITY;
        }
#pragma unroll
        for (int e = 0; e < 16; ++e) mx[e] = max3f(mx[e], max3f(t[e], t[e + 16], t[e + 32]), t[e + 48]);
      }
#pragma unroll
      for (int e = 0; e < 5; ++e) mx[e] = max3f(mx[e], mx[e + 5], mx[e + 10]);
      mx[0] = max3f(max3f(mx[0], mx[1], mx[2]), max3f(mx[3], mx[4], mx[15]), mx[0]);
      const float m = mx[0] * scale_log2;
      // pass 2: P = exp2(s * scale - m) as bf16 pairs over the first half of
      // S (chunk k of 32 keys -> columns 16k .. 16k + 15, already read)
      const unsigned long long sc2 = f2u(scale_log2, scale_log2), nm2 = f2u(-m, -m);
      unsigned long long acc2[4] = {0ull, 0ull, 0ull, 0ull};
      float sq[2][32];
      tmem_ld32_async(s_col, sq[0]);
      tmem_wait32(sq[0]);
      const int nch = 4 * nkv;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (k >= nch) break;
        if (k + 1 < nch) tmem_ld32_async(s_col + (uint32_t)(32 * (k + 1)), sq[(k + 1) & 1]);
        float* x = sq[k & 1];
        const int vt = (k < 4 ? valid0 : valid1) - 32 * (k & 3);
        if (vt < 32) {
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (e >= vt) x[e] = -INFINITY;
        }
        uint32_t pk[16];
        exp_pairs16(x, sc2, nm2, acc2, pk);
        tmem_st16u(s_col + (uint32_t)(16 * k), pk);
        if (k + 1 < nch) tmem_wait32(sq[(k + 1) & 1]);
      }
      const float l = acc_total(acc2);
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(p_ready);
      if (lane == 0) w = wait_a(o_final, it & 1, abort_flag) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
      tc_fence_after();
      // O into registers, then TMEM is released (the next query tile's S
      // MMA may start) before the output is written
      float o[C::DK / 16][16];
#pragma unroll
      for (int c = 0; c < C::DK / 16; ++c) tmem_ld16(o_col + (uint32_t)(c * 16), o[c]);
      tc_fence_before();
      mbar_arrive(o_free);
      const float inv = 1.0f / l;
      bf16* orow = reinterpret_cast<bf16*>(a.out) + (size_t)(qs.row0 + (r < qs.valid ? r : 0)) * a.ld_out + (size_t)h * D;
      if (r < qs.valid) {
#pragma unroll
        for (int c = 0; c < C::DK / 16; ++c) {
#pragma unroll
          for (int e = 0; e < 16; e += 8) {
            if (c * 16 + e < D) {
              float t8[8];
#pragma unroll
              for (int z = 0; z < 8; ++z) t8[z] = o[c][e + z] * inv;
              st16(orow + c * 16 + e, t8);
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
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::TMEM_COLS) : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;
std::once_flag g_once;
int g_attn_sms = 148;

bool init_attn() {
  std::call_once(g_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) == cudaSuccess && cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
        sms > 0)
      g_attn_sms = sms;
#define FF_ATTR(d, qt) \
  cudaFuncSetAttribute(k_attn_tc<d, qt>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ACfg<d, qt>::SMEM)
    FF_ATTR(64, 1); FF_ATTR(64, 2); FF_ATTR(72, 1); FF_ATTR(72, 2); FF_ATTR(128, 1); FF_ATTR(128, 2);
    cudaFuncSetAttribute(k_attn_short<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ShortLayout::SMEM);
    cudaFuncSetAttribute(k_attn_short<72>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ShortLayout::SMEM);
#undef FF_ATTR
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
  // query tiles per sample; short sequences (a few key tiles) run one query
  // tile per CTA, two CTAs per SM, longer ones two query tiles per CTA
  const int nq = (a.Nt + 127) / 128 + (a.Ni + 127) / 128;
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)D);
  if (nq <= 2 && D <= 80) {
    // resident K / V, one N = 256 S per query tile (DiT-XL/2's 256 tokens)
    // q / k columns 64 .. 79 (32-byte swizzle), v in 32-column boxes (64-byte swizzle)
    CUtensorMap tt = tm, tv = tm;
    cuuint32_t box16[3] = {16, 1, 128}, box32[3] = {32, 1, 128};
    if (g_enc(&tt, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.q), dims, strides, box16, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_32B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
        g_enc(&tv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.q), dims, strides, box32, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
    const long long heads = (long long)a.H * a.B, slots = 2LL * g_attn_sms;
    int ipc = 1;
    while (ipc < nq && (long long)((nq + ipc - 1) / ipc) * heads > slots) ++ipc;
    launch_pdl(k_attn_short<D <= 64 ? 64 : 72>, dim3((nq + ipc - 1) / ipc, a.H, a.B), ACfgShort<D <= 64 ? 64 : 72>::THREADS,
               ShortLayout::SMEM, s, tm, tt, tv, a, scale_log2, ipc);
    return launched();
  }
  if (nq <= SHORT_KV_TILES) {
    // query tiles of one (sample, head) per CTA: as few as keep the CTAs
    // within one wave of two per SM, so the second tile's loads overlap the
    // first tile's tail instead of a second wave starting from scratch
    const long long heads = (long long)a.H * a.B, slots = 2LL * g_attn_sms;
    int ipc = 1;
    while (ipc < nq && (long long)((nq + ipc - 1) / ipc) * heads > slots) ++ipc;
    launch_pdl(k_attn_tc<D, 1>, dim3((nq + ipc - 1) / ipc, a.H, a.B), ACfg<D, 1>::THREADS, ACfg<D, 1>::SMEM, s, tm, a,
               scale_log2, ipc);
  } else {
    launch_pdl(k_attn_tc<D, 2>, dim3((nq + 1) / 2, a.H, a.B), ACfg<D, 2>::THREADS, ACfg<D, 2>::SMEM, s, tm, a,
               scale_log2, 1);
  }
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
