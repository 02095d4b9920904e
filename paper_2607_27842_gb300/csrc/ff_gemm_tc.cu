// bf16 dense layers of the exact block (Eq. 1) on the 5th-generation tensor
// cores: out = epilogue(A[M,K] W[N,K]^T).
//
// Persistent kernel, one CTA per SM, 10 warps:
//   warp 0      TMA producer: A and W tiles (128 and BN rows x 64 k, 128-byte
//               swizzle) into a STAGES-deep shared-memory ring;
//   warp 1      TMEM allocator and MMA issuer (the whole warp runs the loop,
//               one elected lane issues):
//               tcgen05.mma.cta_group::1.kind::f16 (M = 128, N = BN, K = 16),
//               fp32 accumulators in TMEM, tcgen05.commit frees ring slots;
//   warps 2..9  epilogue: tcgen05.ld of the accumulator (each warp one
//               32-lane quarter and one column half), the fused bias / RoPE /
//               GELU / gate / residual / history epilogue, stores through
//               swizzled shared-memory blocks and TMA (16-byte stores where
//               the output does not allow it); with one tile per CTA the
//               residual / history-base blocks arrive by TMA as well.
// Two TMEM accumulators (2 * BN columns) let the epilogue of tile i overlap
// the main loop of tile i + 1.  Every mbarrier wait is bounded: on timeout
// the CTA raises a watchdog flag, stops issuing work and releases its TMEM.
//
// With both operands in shared memory a 128 x 128 x 16 MMA is bound by the
// operand reads and takes about as long as a 128 x 256 x 16 one, so narrow
// tiles run at half rate.  With BN = 256 the columns past the last
// full 256-wide tile are covered by swapped tiles: up to 128 rows of W as
// the MMA's M side against 256 rows of A as its N side (the accumulator
// holds the transposed block; the epilogue transposes it back through a
// 16 x 32 shared-memory buffer per warp).  DiT-XL/2's N = 1152 layers then
// run as 4 x 32 full tiles + 16 swapped tiles, one wave of 144 tiles.
#include "ff_common.cuh"
#include "ff_tc.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

namespace ff {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int THREADS = 320;  // producer, MMA, 8 epilogue warps
using namespace tc;

__device__ unsigned int g_watchdog;

__device__ __forceinline__ bool mbar_wait_g(uint64_t* b, uint32_t parity, volatile int* abort_flag) {
  return mbar_wait(b, parity, abort_flag, &g_watchdog);
}
// the producer's waits for a free stage poll: a suspended wait woke up
// several hundred cycles after the stage's MMAs completed, and the ring is
// only four stages deep
__device__ __forceinline__ bool mbar_wait_p(uint64_t* b, uint32_t parity, volatile int* abort_flag) {
  return mbar_wait<true>(b, parity, abort_flag, &g_watchdog);
}
// the MMA warp's waits: every lane waits, the vote keeps the loop control
// (and the descriptors computed under it) warp-uniform, so the elected lane's
// tcgen05.mma does not block the issuing thread
__device__ __forceinline__ bool mbar_wait_u(uint64_t* b, uint32_t parity, volatile int* abort_flag) {
  const bool ok = mbar_test(b, parity) || mbar_wait_g(b, parity, abort_flag);
  return __all_sync(0xffffffffu, ok);
}

template <int BN> struct Cfg {
  static constexpr int STAGES = BN >= 256 ? 4 : 6;
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BYTES = BN * BK * 2;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
  // BN = 256 only: 4 KB per epilogue warp, two 32 x 32 bf16 output blocks
  // for the TMA-store epilogue, or the 16 x 32 fp32 transpose buffer of a
  // swapped tile
  static constexpr uint32_t XPOSE_BYTES = BN >= 256 ? 8 * 4096 : 0;
  static constexpr size_t SMEM = 1024 + (size_t)STAGES * STAGE_BYTES + XPOSE_BYTES + 256;
  // instruction descriptor, kind::f16: D fp32 (bit 4), A bf16 (bits 7-9 = 1),
  // B bf16 (bits 10-12 = 1), both K-major, N >> 3 at bit 17, M >> 4 at bit 24.
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                                    ((uint32_t)(BM >> 4) << 24);
};

// Tile list of one launch: n_norm normal tiles (128 rows of A x BN rows of
// W, M-fastest), then swapped tiles (128 rows of W x 256 rows of A).
struct TileMap {
  int num_m;   // 128-row blocks of A
  int n_full;  // BN-wide column blocks of the normal tiles
  int n_norm;  // num_m * n_full
  int num_m2;  // 256-row blocks of A (swapped tiles)
  int n_tiles; // n_norm + swapped tiles
  int staged;  // normal tiles store out (and hist_out) through shared memory + TMA
  // one tile per CTA (the TMA ring is idle after its mainloop): each
  // epilogue warp loads its residual (bit 0) and history-base (bit 1) block
  // with TMA into the freed ring instead of per-lane global loads
  int pre;
};

// 64-byte-swizzled [32 rows x 32 bf16] block: 16-byte chunk k of row r
__device__ __forceinline__ uint32_t blk_off(int r, int k) { return (uint32_t)(r * 64 + ((k ^ ((r >> 1) & 3)) << 4)); }
__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 t = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&t);
}
__device__ __forceinline__ float2 unpack2(uint32_t u) {
  return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u));
}
struct TileAt {
  bool sw;
  int m0, n0;  // first output row / column
};
template <int BN>
__device__ __forceinline__ TileAt tile_at(const TileMap& t, int tile) {
  if (tile < t.n_norm) return {false, (tile % t.num_m) * BM, (tile / t.num_m) * BN};
  const int u = tile - t.n_norm;
  return {true, (u % t.num_m2) * 256, t.n_full * BN + (u / t.num_m2) * 128};
}

// Per-warp constants of the epilogue warps.
struct EpiWarp {
  uint8_t* smem;      // the 1024-aligned shared-memory base (ring first)
  uint8_t* ep;        // the warp's 4 KB output / transpose buffer
  uint64_t* rbar;     // per-warp residual / history-base barriers
  uint64_t* tfull;    // accumulator-full barriers
  volatile int* abort_flag;
  uint32_t tmem_base;
  int warp, lane, q, h, row, c_lo;
};

// The epilogue of one tile, inlined once per problem of the launch so that
// every EpiArgs / TileMap field and tensor map is read from its own kernel
// parameter (a run-time choice between two parameter structs turns every
// field access of the inner loops into a generic load).  PLAIN: normal
// tiles without residual preloads (the second problem of a grouped launch,
// the CTA pairs).  XB: bytes of the epilogue warps' staging buffers (0: the
// per-lane store path only).  Returns false when the accumulator wait gave up.
template <int BN, int XB, bool PLAIN, int LN>
__device__ __forceinline__ bool epi_tile(const EpiWarp& W, const EpiArgs& e, const TileMap& tm, const int M,
                                         const int N, const TileAt t, const int acc, const uint32_t aph,
                                         uint32_t& epi_cnt, const CUtensorMap* tmO, const CUtensorMap* tmH,
                                         const CUtensorMap* tmR, const CUtensorMap* tmHB) {
  const int warp = W.warp, lane = W.lane, q = W.q, h = W.h, row = W.row, c_lo = W.c_lo;
  uint8_t* const smem = W.smem;
  uint8_t* const ep = W.ep;
  float* const xp = reinterpret_cast<float*>(ep);
  uint64_t* const rbar = W.rbar;
  uint64_t* const tfull = W.tfull;
  volatile int* const abort_flag = W.abort_flag;
  const uint32_t tmem_base = W.tmem_base;
  const int pre = PLAIN ? 0 : tm.pre;
  constexpr int LNM = LN == 1 ? 1 : LN == 2 ? 2 : 0;
  const bool sw = !PLAIN && t.sw;
  uint4 pr[4], ph[4];
  float pb = 0.f, pg0 = 0.f, pg1 = 0.f;
  // staged epilogue: residual / history-base rows of chunk n0 into pr /
  // ph; bias and gate of column n0 + lane into pb / pg0 / pg1 (shared
  // across the warp by shuffles: the warp's 32 rows lie in samples
  // b_lo .. b_hi, at most two of them)
  const int wr0 = t.m0 + q * 32;
  const int b_lo = e.gate ? epi_batch(e, min(wr0, M - 1)) : 0;
  const int b_hi = e.gate ? epi_batch(e, min(wr0 + 31, M - 1)) : 0;
  auto fetch = [&](int n0) {
    const int m = t.m0 + row;
    const bool cin = n0 + lane < N;
    pb = (e.bias && cin) ? __bfloat162float(reinterpret_cast<const bf16*>(e.bias)[n0 + lane]) : 0.f;
    pg0 = (e.gate && cin) ? e.gate[(size_t)b_lo * e.gate_stride + n0 + lane] : 0.f;
    pg1 = (e.gate && cin && b_hi != b_lo) ? e.gate[(size_t)b_hi * e.gate_stride + n0 + lane] : pg0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const bool in = m < M && n0 + 8 * k < N;
      if (e.resid && !(pre & 1))
        pr[k] = in ? *reinterpret_cast<const uint4*>(reinterpret_cast<const bf16*>(e.resid) +
                                                      (size_t)m * e.ld_resid + n0 + 8 * k)
                   : make_uint4(0, 0, 0, 0);
      if (e.hist_out && !(pre & 2))
        ph[k] = in ? *reinterpret_cast<const uint4*>(reinterpret_cast<const bf16*>(e.hist_base) +
                                                      (size_t)m * e.ldo + n0 + 8 * k)
                   : make_uint4(0, 0, 0, 0);
    }
  };
  if (XB > 0 && tm.staged && !sw) fetch(t.n0 + c_lo);
  int ok = 1;
  if (lane == 0) ok = mbar_wait_g(&tfull[acc], aph, abort_flag) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  if (!ok) return false;
  tc_fence_after();
  // One tile per CTA: the ring's last readers (this tile's MMAs) are
  // complete, so the warp's residual / history-base blocks (4 x 32 x 32
  // bf16 each, 64-byte swizzle: the layout of the output blocks) come by
  // TMA into its 8 KB slices of the ring; waited for at first use.
  uint8_t* rsm = smem + (warp - 2) * 8192;
  uint8_t* hsm = smem + 65536 + (warp - 2) * 8192;
  bool pre_wait = pre != 0;
  if (pre && lane == 0) {
    mbar_expect_tx(&rbar[warp - 2], ((pre & 1) ? 8192u : 0u) + ((pre & 2) ? 8192u : 0u));
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int x = sw ? t.n0 + q * 32 : t.n0 + c_lo + 32 * i;
      const int y = sw ? t.m0 + h * (BN / 2) + 32 * i : t.m0 + q * 32;
      if (pre & 1) tma_load(tmR, &rbar[warp - 2], rsm + i * 2048, x, y);
      if (pre & 2) tma_load(tmHB, &rbar[warp - 2], hsm + i * 2048, x, y);
    }
  }
  auto pre_ready = [&]() -> bool {
    if (!pre_wait) return true;
    pre_wait = false;
    int w = 1;
    if (lane == 0) w = mbar_wait_g(&rbar[warp - 2], 0, abort_flag) ? 1 : 0;
    return __shfl_sync(0xffffffffu, w, 0) != 0;
  };
  const uint32_t tq = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
  if (!sw && (XB == 0 || !tm.staged)) {
    const int m = t.m0 + row;
    const float2 lnr = ((LN == 1 && e.ln_in) && m < M) ? ln_row(e, m) : make_float2(1.f, 0.f);
    for (int c = h * (BN / 2); c < (h + 1) * (BN / 2); c += 32) {
      const int n0 = t.n0 + c;
      if (n0 >= N) break;
      float v[32];
      tmem_ld32(tq + (uint32_t)c, v);
      if (m < M) {
        const float2 st = epi_chunk<bf16, 32, LNM>(e, m, n0, N, v, lnr);
        if ((LN == 2 && e.ln_out)) ln_put(e, m, n0, st);
      }
    }
  } else if (!sw) {
    // Staged epilogue: each 32-row x 32-column chunk is written into a
    // swizzled shared-memory block and stored by one TMA copy (whole
    // lines instead of one L2 request per 16 bytes).  The residual and
    // history-base rows of a chunk are loaded ahead: the first chunk's
    // before the accumulator wait, the next one's while the current
    // chunk is finished.
    const int m = t.m0 + row;
    const int bm = m < M ? epi_batch(e, m) : 0;   // the row's sample (fused LayerNorm)
    const float2 lnr = ((LN == 1 && e.ln_in) && m < M) ? ln_row(e, m) : make_float2(1.f, 0.f);
    for (int c = c_lo; c < c_lo + BN / 2; c += 32) {
      const int n0 = t.n0 + c;
      if (n0 >= N) break;
      float v[32];
      tmem_ld32(tq + (uint32_t)c, v);
      // y = gate * act(rope(acc + bias)), the order of epi_math; rows
      // past M are not stored (the TMA store clips them)
      if ((LN == 1 && e.ln_in) && m < M) ln_correct<32>(e, bm, n0, N, lnr, v);
      if (e.bias) {
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] += __shfl_sync(0xffffffffu, pb, j);
      }
      if (m < M) epi_rope_act<bf16, 32>(e, m, n0, v);
      if (e.gate) {
        if (b_hi == b_lo) {  // the warp's rows in one sample: one gate row (warp-uniform)
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] *= __shfl_sync(0xffffffffu, pg0, j);
        } else {
          const bool lo = m >= M || epi_batch(e, m) == b_lo;
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float g0 = __shfl_sync(0xffffffffu, pg0, j), g1 = __shfl_sync(0xffffffffu, pg1, j);
            v[j] *= lo ? g0 : g1;
          }
        }
      }
      if (pre) {
        if (!pre_ready()) { ok = 0; break; }
        const uint8_t* rb = rsm + ((c - c_lo) >> 5) * 2048;
        const uint8_t* hb2 = hsm + ((c - c_lo) >> 5) * 2048;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if (pre & 1) pr[k] = *reinterpret_cast<const uint4*>(rb + blk_off(lane, k));
          if (pre & 2) ph[k] = *reinterpret_cast<const uint4*>(hb2 + blk_off(lane, k));
        }
      }
      uint32_t ob[16], hb[16];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t rr[4] = {pr[k].x, pr[k].y, pr[k].z, pr[k].w};
        const uint32_t hh[4] = {ph[k].x, ph[k].y, ph[k].z, ph[k].w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          float a = v[8 * k + 2 * i], b = v[8 * k + 2 * i + 1];
          if (e.resid) {
            const float2 r2 = unpack2(rr[i]);
            a += r2.x;
            b += r2.y;
          }
          ob[4 * k + i] = pack2(a, b);
          if (e.hist_out) {  // stored(out) - hist_base
            const float2 o2 = unpack2(ob[4 * k + i]), h2 = unpack2(hh[i]);
            hb[4 * k + i] = pack2(o2.x - h2.x, o2.y - h2.y);
          }
        }
      }
      if ((LN == 2 && e.ln_out) && m < M) {  // the next layer's scaled copy and chunk statistics
        float x[32];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const float2 f = unpack2(ob[k]);
          x[2 * k] = f.x;
          x[2 * k + 1] = f.y;
        }
        ln_put(e, m, n0, ln_emit<32>(e, m, bm, n0, x));
      }
      if (c + 32 < c_lo + BN / 2 && n0 + 32 < N) fetch(n0 + 32);
      // block(s) for this chunk: out alternates between the two when
      // there is no history stream, else out -> block 0, hist -> block 1
      uint8_t* b0 = ep + (e.hist_out ? 0 : (epi_cnt & 1) * 2048);
      if (lane == 0) {
        if (e.hist_out) bulk_wait_read<0>(); else bulk_wait_read<1>();
      }
      __syncwarp();
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        *reinterpret_cast<uint4*>(b0 + blk_off(lane, k)) = make_uint4(ob[4 * k], ob[4 * k + 1], ob[4 * k + 2], ob[4 * k + 3]);
        if (e.hist_out)
          *reinterpret_cast<uint4*>(ep + 2048 + blk_off(lane, k)) =
              make_uint4(hb[4 * k], hb[4 * k + 1], hb[4 * k + 2], hb[4 * k + 3]);
      }
      fence_async_smem();
      __syncwarp();
      if (lane == 0) {
        tma_store(tmO, b0, n0, t.m0 + q * 32);
        if (e.hist_out) tma_store(tmH, ep + 2048, n0, t.m0 + q * 32);
        bulk_commit();
      }
      ++epi_cnt;
    }
  } else if constexpr (XB > 0) {
    // lane = output column n + lane; TMEM column = output row.  Blocks of
    // 16 rows x 32 columns go through the warp's buffer (XOR-swizzled,
    // conflict-free both ways); afterwards lane l holds row l / 2,
    // columns 16 (l % 2) .. + 15.
    const int n = t.n0 + q * 32;
    if (lane == 0) bulk_wait_read<0>();  // TMA stores of earlier tiles done reading the buffer
    __syncwarp();
    // preloaded form: the lane's 16 columns are the same for every block
    // of rows, so their bias stays in registers and the gate row is
    // reloaded only when the row's sample changes
    const bool pre_sw = pre && !e.out_f32 && e.split_col >= N && !e.rope;
    float bv[16], gv[16];
    int gb = -1;
    if (pre_sw) {
      const int nc0 = n + (lane & 1) * 16;
#pragma unroll
      for (int g = 0; g < 2; ++g) {
        float b8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        if (e.bias && nc0 + 8 * g < N) ld16(reinterpret_cast<const bf16*>(e.bias) + nc0 + 8 * g, b8);
#pragma unroll
        for (int k = 0; k < 8; ++k) bv[8 * g + k] = b8[k];
      }
    }
    for (int c = h * (BN / 2); c < (h + 1) * (BN / 2) && n < N; c += 16) {
      const int m0 = t.m0 + c;
      if (m0 >= M) break;
      {
        float u[16];
        tmem_ld16(tq + (uint32_t)c, u);  // u[j] = out[m0 + j][n + lane]
#pragma unroll
        for (int j = 0; j < 16; ++j) xp[j * 32 + (lane ^ j)] = u[j];
      }
      __syncwarp();
      const int r = lane >> 1, c0 = (lane & 1) * 16;
      float v[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) v[j] = xp[r * 32 + ((c0 + j) ^ r)];  // out[m0 + r][n + c0 + j]
      __syncwarp();
      const int m = m0 + r;
      if (pre && !e.out_f32 && e.split_col >= N) {
        // residual / history base of row m from the warp's ring slices
        // (block (row in the warp's 128 rows) / 32, 16-byte chunks
        // c0 / 8 and c0 / 8 + 1 of that row)
        if (!pre_ready()) break;
        float2 lst = make_float2(0.f, 0.f);   // fused LayerNorm: this lane's 16-column statistics
        if (m < M) {
          if (pre_sw) {  // epi_math's order: act(acc + bias) * gate
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] += bv[j];
            epi_rope_act<bf16, 16>(e, m, n + c0, v);
            if (e.gate) {
              const int bt = epi_batch(e, m);
              if (bt != gb) {
                gb = bt;
                const float* gp = e.gate + (size_t)bt * e.gate_stride + n + c0;
#pragma unroll
                for (int j = 0; j < 16; j += 4) {
                  const float4 g4 = n + c0 + j < N ? *reinterpret_cast<const float4*>(gp + j)
                                                   : make_float4(0.f, 0.f, 0.f, 0.f);
                  gv[j] = g4.x; gv[j + 1] = g4.y; gv[j + 2] = g4.z; gv[j + 3] = g4.w;
                }
              }
#pragma unroll
              for (int j = 0; j < 16; ++j) v[j] *= gv[j];
            }
          } else {
            epi_math<bf16, 16, LNM>(e, m, n + c0, N, v);
          }
          const int rw = c - h * (BN / 2) + r;
          const uint32_t base = (uint32_t)((rw >> 5) * 2048);
          float xs[16];   // stored values of the lane's 16 columns
#pragma unroll
          for (int j = 0; j < 16; ++j) xs[j] = 0.f;
#pragma unroll
          for (int g = 0; g < 2; ++g) {
            const int nc = n + c0 + 8 * g;
            if (nc >= N) continue;
            const uint32_t off = base + blk_off(rw & 31, (c0 >> 3) + g);
            uint4 rv = make_uint4(0, 0, 0, 0), hv = make_uint4(0, 0, 0, 0);
            if (pre & 1)
              rv = *reinterpret_cast<const uint4*>(rsm + off);
            else if (e.resid)
              rv = *reinterpret_cast<const uint4*>(reinterpret_cast<const bf16*>(e.resid) + (size_t)m * e.ld_resid + nc);
            if (e.hist_out)
              hv = (pre & 2) ? *reinterpret_cast<const uint4*>(hsm + off)
                                : *reinterpret_cast<const uint4*>(reinterpret_cast<const bf16*>(e.hist_base) +
                                                                  (size_t)m * e.ldo + nc);
            const uint32_t rr4[4] = {rv.x, rv.y, rv.z, rv.w}, hh4[4] = {hv.x, hv.y, hv.z, hv.w};
            uint32_t ob[4], hb[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              float a = v[8 * g + 2 * i], b = v[8 * g + 2 * i + 1];
              if (e.resid) {
                const float2 r2 = unpack2(rr4[i]);
                a += r2.x;
                b += r2.y;
              }
              ob[i] = pack2(a, b);
              const float2 o2 = unpack2(ob[i]);
              xs[8 * g + 2 * i] = o2.x;
              xs[8 * g + 2 * i + 1] = o2.y;
              if (e.hist_out) {  // stored(out) - hist_base
                const float2 h2 = unpack2(hh4[i]);
                hb[i] = pack2(o2.x - h2.x, o2.y - h2.y);
              }
            }
            *reinterpret_cast<uint4*>(reinterpret_cast<bf16*>(e.out) + (size_t)m * e.ldo + nc) =
                make_uint4(ob[0], ob[1], ob[2], ob[3]);
            if (e.hist_out)
              *reinterpret_cast<uint4*>(reinterpret_cast<bf16*>(e.hist_out) + (size_t)m * e.ldo + nc) =
                  make_uint4(hb[0], hb[1], hb[2], hb[3]);
          }
          if ((LN == 2 && e.ln_out)) lst = ln_emit<16>(e, m, epi_batch(e, m), n + c0, xs);
        }
        if ((LN == 2 && e.ln_out)) {  // lanes l and l ^ 1 hold the two halves of the row's 32 columns
          lst = ln_pair(lst);
          if (!(lane & 1) && m < M) ln_put(e, m, n, lst);
        }
        continue;
      }
      float2 lst = make_float2(0.f, 0.f);
      if (m < M) lst = epi_chunk<bf16, 16, LNM>(e, m, n + c0, N, v, (LN == 1 && e.ln_in) ? ln_row(e, m) : make_float2(1.f, 0.f));
      if ((LN == 2 && e.ln_out)) {
        lst = ln_pair(lst);
        if (!(lane & 1) && m < M) ln_put(e, m, n, lst);
      }
    }
  }
  // a warp whose columns all lie past N never read its blocks: their
  // copies still land before it moves on
  if (pre_wait) pre_ready();
  return true;
}

// GROUPED: a second problem (group 1, tm1.n_tiles > 0) of the same N and K
// with its own A, W, rows and epilogue (the text stream of a two-stream
// block beside the image stream), its tiles first in the tile list; both
// groups then have only normal tiles and no residual preloads.  Without
// GROUPED the group-1 parameters are unused.
template <int BN, bool GROUPED, int LN>
__global__ void __launch_bounds__(THREADS, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
              const __grid_constant__ CUtensorMap tmW128, const __grid_constant__ CUtensorMap tmA256,
              const __grid_constant__ CUtensorMap tmO, const __grid_constant__ CUtensorMap tmH,
              const __grid_constant__ CUtensorMap tmR, const __grid_constant__ CUtensorMap tmHB, int M0, int N, int K,
              const __grid_constant__ TileMap tm0, const __grid_constant__ EpiArgs e0,
              const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
              const __grid_constant__ CUtensorMap tmO1, const __grid_constant__ CUtensorMap tmH1, int M1,
              const __grid_constant__ TileMap tm1, const __grid_constant__ EpiArgs e1) {
  using C = Cfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  float* xpose = reinterpret_cast<float*>(sB + C::STAGES * C::B_BYTES);
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + C::STAGES * C::B_BYTES + C::XPOSE_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* rbar = tempty + 2;  // per epilogue warp: its residual / history-base blocks landed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(rbar + 8);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n1 = GROUPED ? tm1.n_tiles : 0;
  const int num_tiles = tm0.n_tiles + n1;
  const int num_kb = (K + BK - 1) / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 256);
    }
    for (int w = 0; w < 8; ++w) mbar_init(&rbar[w], 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmA) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmB) : "memory");
    if (tm0.pre & 1) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmR) : "memory");
    if (tm0.pre & 2) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmHB) : "memory");
    if (GROUPED && n1) {
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmA1) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmB1) : "memory");
    }
    if (tm0.n_tiles > tm0.n_norm) {
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmW128) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmA256) : "memory");
    }
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
  const uint32_t tmem_base = *tmem_slot;
  // dependents may launch once every CTA holds its TMEM; the previous
  // kernel's outputs are complete after the wait
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        const bool g1 = GROUPED && tile < n1;
        const TileAt t = g1 ? tile_at<BN>(tm1, tile) : tile_at<BN>(tm0, tile - n1);
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % C::STAGES;
          const uint32_t ph = (it / C::STAGES) & 1;
          if (!mbar_wait_p(&empty[s], ph ^ 1, abort_flag)) { ok = false; break; }
          mbar_expect_tx(&full[s], C::STAGE_BYTES);
          // normal: A rows -> M side, W rows -> N side; swapped: the reverse.
          // (Each call names its kernel parameter: a tensor map must stay in
          // parameter space, never be copied to local memory.)
          if (g1) {
            tma_load(&tmA1, &full[s], sA + s * C::A_BYTES, kb * BK, t.m0);
            tma_load(&tmB1, &full[s], sB + s * C::B_BYTES, kb * BK, t.n0);
          } else if (!t.sw) {
            tma_load(&tmA, &full[s], sA + s * C::A_BYTES, kb * BK, t.m0);
            tma_load(&tmB, &full[s], sB + s * C::B_BYTES, kb * BK, t.n0);
          } else {
            tma_load(&tmW128, &full[s], sA + s * C::A_BYTES, kb * BK, t.n0);
            tma_load(&tmA256, &full[s], sB + s * C::B_BYTES, kb * BK, t.m0);
          }
        }
      }
      // Copies still in flight complete on their full barriers; wait for
      // the last ring's worth so none lands after the CTA exits.
      for (uint32_t k = 0; k < (uint32_t)C::STAGES && k < it; ++k) {
        const uint32_t j = it - 1 - k;
        const unsigned long long t0 = gtimer();
        while (!mbar_try(&full[j % C::STAGES], (j / C::STAGES) & 1)) {
          if (gtimer() - t0 > WAIT_LIMIT_NS) { atomicOr(&g_watchdog, 2u); break; }
        }
      }
    }
  } else if (warp == 1) {
    // the whole warp runs the loop, one elected lane issues
    uint32_t it = 0;
    int tc = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x, ++tc) {
      const int acc = tc & 1;
      const uint32_t aph = (tc >> 1) & 1;
      if (!mbar_wait_u(&tempty[acc], aph ^ 1, abort_flag)) break;
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
      for (int kb = 0; kb < num_kb; ++kb, ++it) {
        const int s = it % C::STAGES;
        const uint32_t ph = (it / C::STAGES) & 1;
        if (!mbar_wait_u(&full[s], ph, abort_flag)) { ok = false; break; }
        tc_fence_after();
        const uint64_t ad = sw128_desc(saddr(sA + s * C::A_BYTES));
        const uint64_t bd = sw128_desc(saddr(sB + s * C::B_BYTES));
#pragma unroll
        for (int k = 0; k < BK / 16; ++k) {
          // +32 bytes (16 bf16) along K inside the swizzle atom
          if (elect_one()) umma(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), C::IDESC, (kb | k) != 0);
        }
        if (elect_one()) umma_commit(&empty[s]);
      }
      if (!ok) break;
      if (elect_one()) umma_commit(&tfull[acc]);
    }
  } else {
    // 8 epilogue warps: TMEM lane quarter q = warp % 4 (the quarter a warp
    // may access), column half h of the tile
    const int q = warp & 3;
    const int h = (warp - 2) >> 2;
    const EpiWarp W = {smem, reinterpret_cast<uint8_t*>(xpose) + (warp - 2) * 4096, rbar, tfull, abort_flag,
                       tmem_base, warp, lane, q, h, q * 32 + lane, h * (BN / 2)};
    int tc = 0;
    uint32_t epi_cnt = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++tc) {
      const int acc = tc & 1;
      const uint32_t aph = (tc >> 1) & 1;
      bool ok;
      if constexpr (GROUPED) {
        ok = tile < n1 ? epi_tile<BN, Cfg<BN>::XPOSE_BYTES, true, LN>(W, e1, tm1, M1, N, tile_at<BN>(tm1, tile), acc, aph, epi_cnt, &tmO1,
                                            &tmH1, &tmR, &tmHB)
                       : epi_tile<BN, Cfg<BN>::XPOSE_BYTES, true, LN>(W, e0, tm0, M0, N, tile_at<BN>(tm0, tile - n1), acc, aph, epi_cnt, &tmO,
                                            &tmH, &tmR, &tmHB);
      } else {
        ok = epi_tile<BN, Cfg<BN>::XPOSE_BYTES, false, LN>(W, e0, tm0, M0, N, tile_at<BN>(tm0, tile), acc, aph, epi_cnt, &tmO, &tmH, &tmR,
                                 &tmHB);
      }
      if (!ok) break;
      tc_fence_before();
      mbar_arrive(&tempty[acc]);
    }
    if (C::XPOSE_BYTES > 0 && lane == 0) bulk_wait_all();  // TMA stores complete before exit
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(C::TMEM_COLS)
                 : "memory");
  }
}

// ---------------------------------------------------------------------------
// CTA-pair variant: a cluster of 2 CTAs computes a 256 x BN tile with
// tcgen05.mma.cta_group::2 (M = 256).  Each CTA stages its own 128 rows of A
// and half (BN/2 rows) of W, so per CTA the shared-memory traffic per FLOP
// is that of a 128 x 2BN tile.  The even CTA issues the MMAs; its full
// barriers collect both CTAs' TMA bytes; commits are multicast to both CTAs'
// empty / accumulator-full barriers; both CTAs' epilogues arrive on the even
// CTA's accumulator-empty barrier.
// ---------------------------------------------------------------------------
template <int BN> struct Cfg2 {
  static constexpr int HB = BN / 2;
  static constexpr int STAGES = BN >= 256 ? 6 : 8;
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BYTES = HB * BK * 2;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
  static constexpr uint32_t XPOSE_BYTES = 8 * 4096;  // the staged epilogue's output blocks
  static constexpr size_t SMEM = 1024 + (size_t)STAGES * STAGE_BYTES + XPOSE_BYTES + 256;
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                                    ((uint32_t)(256 >> 4) << 24);
};

// The epilogue is epi_tile's (staged TMA-store blocks where tm.staged), each
// CTA on its own 128 rows of the pair's 256-row tile.
// GROUPED: a second problem of the same N and K (its own A, W, rows,
// epilogue and store maps: the text stream of a two-stream block beside the
// image stream), its tiles first in the tile list, so its few tiles fill the
// first problem's last wave instead of running alone on a handful of SMs.
template <int BN, int LN, bool GROUPED>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
    k_gemm_tc2(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               const __grid_constant__ CUtensorMap tmO, const __grid_constant__ CUtensorMap tmH, int M, int N, int K,
               const __grid_constant__ TileMap tm, const __grid_constant__ EpiArgs e,
               const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
               const __grid_constant__ CUtensorMap tmO1, const __grid_constant__ CUtensorMap tmH1, int M1,
               const __grid_constant__ TileMap tm1, const __grid_constant__ EpiArgs e1) {
  using C = Cfg2<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint8_t* xpose = sB + C::STAGES * C::B_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(xpose + C::XPOSE_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  const int num_m = (M + 2 * BM - 1) / (2 * BM), num_n = (N + BN - 1) / BN;
  const int num_m1 = GROUPED ? (M1 + 2 * BM - 1) / (2 * BM) : 0;
  const int n1 = num_m1 * num_n;              // group 1's tiles come first
  const int num_tiles = n1 + num_m * num_n;
  // (group, row block, column block) of tile `tile`
  auto tile_of = [&](int tile, bool& g1, int& mb, int& nb) {
    g1 = GROUPED && tile < n1;
    const int u = g1 ? tile : tile - n1;
    const int nm = g1 ? num_m1 : num_m;
    mb = u % nm;
    nb = u / nm;
  };
  const int num_kb = (K + BK - 1) / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 2 * 256);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmA) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmB) : "memory");
    if (GROUPED && n1) {
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmA1) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmB1) : "memory");
    }
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(tmem_slot)),
                 "r"(C::TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncwarp();
  cluster_sync_all();  // both CTAs' barriers initialised before any cross-CTA use
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // dependents may launch once every CTA holds its TMEM; the previous
  // kernel's outputs are complete after the wait
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += npairs) {
        bool g1;
        int mb, nb;
        tile_of(tile, g1, mb, nb);
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % C::STAGES;
          const uint32_t ph = (it / C::STAGES) & 1;
          if (!mbar_wait_p(&empty[s], ph ^ 1, abort_flag)) { ok = false; break; }
          if (leader) mbar_expect_tx(&full[s], 2 * C::STAGE_BYTES);
          const uint32_t fb = map_to(&full[s], 0);
          // (each call names its kernel parameter: a tensor map stays in
          // parameter space)
          if (g1) {
            tma_load_pair(&tmA1, fb, sA + s * C::A_BYTES, kb * BK, mb * 2 * BM + (int)rank * BM);
            tma_load_pair(&tmB1, fb, sB + s * C::B_BYTES, kb * BK, nb * BN + (int)rank * C::HB);
          } else {
            tma_load_pair(&tmA, fb, sA + s * C::A_BYTES, kb * BK, mb * 2 * BM + (int)rank * BM);
            tma_load_pair(&tmB, fb, sB + s * C::B_BYTES, kb * BK, nb * BN + (int)rank * C::HB);
          }
        }
      }
      if (leader) {  // the even CTA's full barriers track both CTAs' copies
        for (uint32_t k = 0; k < (uint32_t)C::STAGES && k < it; ++k) {
          const uint32_t j = it - 1 - k;
          const unsigned long long t0 = gtimer();
          while (!mbar_try(&full[j % C::STAGES], (j / C::STAGES) & 1)) {
            if (gtimer() - t0 > WAIT_LIMIT_NS) { atomicOr(&g_watchdog, 2u); break; }
          }
        }
      }
    }
  } else if (warp == 1) {
    if (leader) {  // the whole warp runs the loop, one elected lane issues
      uint32_t it = 0;
      int tc = 0;
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += npairs, ++tc) {
        const int acc = tc & 1;
        const uint32_t aph = (tc >> 1) & 1;
        if (!mbar_wait_u(&tempty[acc], aph ^ 1, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % C::STAGES;
          const uint32_t ph = (it / C::STAGES) & 1;
          if (!mbar_wait_u(&full[s], ph, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint64_t ad = sw128_desc(saddr(sA + s * C::A_BYTES));
          const uint64_t bd = sw128_desc(saddr(sB + s * C::B_BYTES));
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            if (elect_one()) umma_pair(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), C::IDESC, (kb | k) != 0);
          if (elect_one()) umma_commit_pair(&empty[s]);
        }
        if (!ok) break;
        if (elect_one()) umma_commit_pair(&tfull[acc]);
      }
    }
  } else {
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int h = (warp - 2) >> 2;  // column half of the tile
    const EpiWarp W = {smem, xpose + (warp - 2) * 4096, tfull, tfull, abort_flag, tmem_base, warp, lane, q, h,
                       q * 32 + lane, h * (BN / 2)};
    int tc = 0;
    uint32_t epi_cnt = 0;
    for (int tile = pair; tile < num_tiles; tile += npairs, ++tc) {
      bool g1;
      int mb, nb;
      tile_of(tile, g1, mb, nb);
      const int acc = tc & 1;
      const uint32_t aph = (tc >> 1) & 1;
      const TileAt t = {false, mb * 2 * BM + (int)rank * BM, nb * BN};
      bool ok;
      if (g1)
        ok = epi_tile<BN, C::XPOSE_BYTES, true, LN>(W, e1, tm1, M1, N, t, acc, aph, epi_cnt, &tmO1, &tmH1, &tmO1,
                                                     &tmO1);
      else
        ok = epi_tile<BN, C::XPOSE_BYTES, true, LN>(W, e, tm, M, N, t, acc, aph, epi_cnt, &tmO, &tmH, &tmO, &tmO);
      if (!ok) break;
      tc_fence_before();
      mbar_arrive_cluster(map_to(&tempty[acc], 0));
    }
    if (lane == 0) bulk_wait_all();  // TMA stores complete before exit
  }
  tc_fence_before();
  __syncwarp();
  cluster_sync_all();  // no CTA leaves while its peer may still address its TMEM or barriers
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(C::TMEM_COLS)
                 : "memory");
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
// k_gemm_tc instance for a fused-LayerNorm side (0 none, 1 consumer, 2 producer)
template <int BN, bool G>
auto gemm_fn(int ln) -> decltype(&k_gemm_tc<BN, G, 0>) {
  return ln == 1 ? k_gemm_tc<BN, G, 1> : ln == 2 ? k_gemm_tc<BN, G, 2> : k_gemm_tc<BN, G, 0>;
}
template <int BN, bool G = false>
auto gemm2_fn(int ln) -> decltype(&k_gemm_tc2<BN, 0, G>) {
  return ln == 1 ? k_gemm_tc2<BN, 1, G> : ln == 2 ? k_gemm_tc2<BN, 2, G> : k_gemm_tc2<BN, 0, G>;
}
int ln_side(const EpiArgs& e) { return e.ln_in ? 1 : e.ln_out ? 2 : 0; }
// a fused LayerNorm side: one side per launch, bf16 output of whole
// 32-column chunks for the producer, 16-byte aligned rows everywhere
bool ln_ok(const EpiArgs& e, int N) {
  if (e.ln_in && e.ln_out) return false;
  if (e.ln_out && (e.out_f32 || N % 32 != 0 || e.split_col < N || e.ldo % 8 != 0 || !e.ln_scale || !e.ln_stats ||
                   e.ln_stride % 4 != 0 || ((uintptr_t)e.ln_scale & 15) || ((uintptr_t)e.ln_out & 15) ||
                   e.ln_slots * 32 < N))
    return false;
  if (e.ln_in && (!e.ln_c || !e.ln_d || e.ln_cols <= 0 || e.ln_slots * 32 != e.ln_cols || (e.ln_slots & 1) ||
                  e.ln_cd_stride % 4 != 0 ||
                  ((uintptr_t)e.ln_c & 15) || ((uintptr_t)e.ln_d & 15) || ((uintptr_t)e.ln_in & 15)))
    return false;
  return true;
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_once;
int g_sms = 0;

bool init_driver() {
  std::call_once(g_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev);
    if (g_sms <= 0) g_sms = 148;
    for (int ln = 0; ln < 3; ++ln) {
      cudaFuncSetAttribute(gemm_fn<128, false>(ln), cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<128>::SMEM);
      cudaFuncSetAttribute(gemm_fn<256, false>(ln), cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<256>::SMEM);
      cudaFuncSetAttribute(gemm_fn<256, true>(ln), cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg<256>::SMEM);
    }
    for (int ln = 0; ln < 3; ++ln) {
      cudaFuncSetAttribute(gemm2_fn<128>(ln), cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg2<128>::SMEM);
      cudaFuncSetAttribute(gemm2_fn<256>(ln), cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg2<256>::SMEM);
      cudaFuncSetAttribute(gemm2_fn<128, true>(ln), cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg2<128>::SMEM);
      cudaFuncSetAttribute(gemm2_fn<256, true>(ln), cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg2<256>::SMEM);
    }
  });
  return g_encode != nullptr;
}

// 2-D bf16 tensor map over a row-major [rows, cols] matrix with row stride
// ld elements, box [box_rows, 64], 128-byte swizzle, zero fill out of bounds.
bool make_map(CUtensorMap* m, const void* base, int rows, int cols, int ld, int box_rows) {
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Store map of the staged epilogue: [rows, cols] bf16 with row stride ld
// elements, box 32 x 32, 64-byte swizzle (one block row = 64 bytes).
bool make_store_map(CUtensorMap* m, void* base, int rows, int cols, int ld) {
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// The staged (TMA-store) epilogue: one bf16 output of 16-byte aligned rows,
// plus the history stream when present, and a warp's 32 rows spanning at
// most two gate rows.  Encodes the store maps; false where the per-lane
// store path has to be used.
bool staged_maps(const EpiArgs& e, int M, int N, CUtensorMap* mo, CUtensorMap* mh) {
  const bool aligned = !((uintptr_t)e.out & 15) && e.ldo % 8 == 0 &&
                       (!e.hist_out || (!((uintptr_t)e.hist_out & 15) && !((uintptr_t)e.hist_base & 15)));
  const bool gate_ok = !e.gate || ((e.seg_split <= 0 || e.rpb0 >= 32) && e.rpb1 >= 32);
  return !e.out_f32 && e.split_col >= N && aligned && gate_ok && make_store_map(mo, e.out, M, N, e.ldo) &&
         (!e.hist_out || make_store_map(mh, e.hist_out, M, N, e.ldo));
}

// Tile width choice: the fewest waves of rows_per_tile x BN tiles over the
// available CTAs (or CTA pairs), ties to the wider tile (less shared-memory
// traffic per FLOP).
int pick_bn(int M, int N, int rows_per_tile, int slots) {
  double best = 1e30;
  int bn = 256;
  for (int cand : {256, 128}) {
    const long long tiles = (long long)((M + rows_per_tile - 1) / rows_per_tile) * ((N + cand - 1) / cand);
    const long long waves = (tiles + slots - 1) / slots;
    const double cost = (double)waves * cand;
    if (cost < best - 1e-9) { best = cost; bn = cand; }
  }
  return bn;
}

}  // namespace

cudaError_t gemm_tc(int M, int N, int K, const void* A, int lda, const void* W, int ldw, const EpiArgs& e,
                    cudaStream_t s) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  if (!init_driver()) return cudaErrorNotSupported;
  if (K % 8 != 0 || lda % 8 != 0 || ldw % 8 != 0 || N % 8 != 0) return cudaErrorInvalidValue;
  if (!ln_ok(e, N)) return cudaErrorInvalidValue;
  if (((uintptr_t)A & 15) || ((uintptr_t)W & 15)) return cudaErrorInvalidValue;
  CUtensorMap ma, mb;
  // Long reductions: CTA pairs (256-row tiles, each CTA stages half of W);
  // measured faster than single CTAs only from K of about 8k on.  (256 x 128
  // pair tiles for the one-wave DiT-XL/2 layers, two tiles per pair so that
  // an epilogue runs beside the next mainloop, measured slower: fc2 44.8 ->
  // 49.8 us, out-projection 19.1 -> 18.0 us.)
  if (M >= 2 * BM && K >= 8192) {
    const int pairs = g_sms / 2;
    const int bn = pick_bn(M, N, 2 * BM, pairs);
    if (!make_map(&ma, A, M, K, lda, BM) || !make_map(&mb, W, N, K, ldw, bn / 2)) return cudaErrorInvalidValue;
    const long long tiles = (long long)((M + 2 * BM - 1) / (2 * BM)) * ((N + bn - 1) / bn);
    const int grid = 2 * (int)(tiles < pairs ? tiles : pairs);
    TileMap tm2 = {};
    CUtensorMap mo = ma, mh = ma;
    tm2.staged = staged_maps(e, M, N, &mo, &mh) ? 1 : 0;
    const TileMap none = {};
    if (bn == 256)
      launch_pdl(gemm2_fn<256>(ln_side(e)), grid, THREADS, Cfg2<256>::SMEM, s, ma, mb, mo, mh, M, N, K, tm2, e, ma, mb,
                 mo, mh, 0, none, e);
    else
      launch_pdl(gemm2_fn<128>(ln_side(e)), grid, THREADS, Cfg2<128>::SMEM, s, ma, mb, mo, mh, M, N, K, tm2, e, ma, mb,
                 mo, mh, 0, none, e);
    return launched();
  }
  // Every tile (128 x 256 full rate, 128 x 128 at half rate, swapped 128 x
  // 256) takes about the same time: take the tiling with the fewest waves,
  // ties to full-rate tiles.
  TileMap tm;
  tm.num_m = (M + BM - 1) / BM;
  tm.num_m2 = (M + 255) / 256;
  const int rem = N % 256;
  const long long t256 = (long long)tm.num_m * (N / 256) + (rem ? (long long)((rem + 127) / 128) * tm.num_m2 : 0);
  const long long t128 = (long long)tm.num_m * ((N + 127) / 128);
  const bool wide = (t256 + g_sms - 1) / g_sms <= (t128 + g_sms - 1) / g_sms;
  CUtensorMap mw128 = {}, ma256 = {}, mo = {}, mh = {}, mr = {}, mhb = {};
  tm.staged = 0;
  tm.pre = 0;
  if (wide) {
    tm.n_full = N / 256;
    tm.n_norm = tm.num_m * tm.n_full;
    tm.n_tiles = (int)t256;
    if (!make_map(&ma, A, M, K, lda, BM) || !make_map(&mb, W, N, K, ldw, 256)) return cudaErrorInvalidValue;
    if (rem && (!make_map(&mw128, W, N, K, ldw, BM) || !make_map(&ma256, A, M, K, lda, 256)))
      return cudaErrorInvalidValue;
    // staged (TMA-store) epilogue: one bf16 output of 16-byte aligned rows,
    // plus the history stream when present
    const bool aligned = !((uintptr_t)e.out & 15) && e.ldo % 8 == 0 &&
                         (!e.hist_out || (!((uintptr_t)e.hist_out & 15) && !((uintptr_t)e.hist_base & 15)));
    // (a warp's 32 rows must span at most two gate rows)
    const bool gate_ok = !e.gate || ((e.seg_split <= 0 || e.rpb0 >= 32) && e.rpb1 >= 32);
    if (!e.out_f32 && e.split_col >= N && aligned && gate_ok && make_store_map(&mo, e.out, M, N, e.ldo) &&
        (!e.hist_out || make_store_map(&mh, e.hist_out, M, N, e.ldo)))
      tm.staged = 1;
    // one tile per CTA: residual / history-base blocks by TMA into the idle
    // ring (16-byte aligned rows; otherwise the per-lane loads stay)
    if (tm.staged && t256 <= g_sms) {
      if (e.resid && make_store_map(&mr, const_cast<void*>(e.resid), M, N, e.ld_resid)) tm.pre |= 1;
      if (e.hist_out && make_store_map(&mhb, const_cast<void*>(e.hist_base), M, N, e.ldo)) tm.pre |= 2;
    }
    const int grid = (int)(t256 < g_sms ? t256 : g_sms);
    const TileMap none = {};
    launch_pdl(gemm_fn<256, false>(ln_side(e)), grid, THREADS, Cfg<256>::SMEM, s, ma, mb, mw128, ma256, mo, mh, mr, mhb, M, N, K, tm,
               e, ma, mb, mo, mh, 0, none, e);
  } else {
    tm.n_full = (N + 127) / 128;
    tm.n_norm = tm.num_m * tm.n_full;
    tm.n_tiles = tm.n_norm;
    if (!make_map(&ma, A, M, K, lda, BM) || !make_map(&mb, W, N, K, ldw, 128)) return cudaErrorInvalidValue;
    const int grid = (int)(t128 < g_sms ? t128 : g_sms);
    const TileMap none = {};
    launch_pdl(gemm_fn<128, false>(ln_side(e)), grid, THREADS, Cfg<128>::SMEM, s, ma, mb, ma, mb, ma, mb, ma, mb, M, N, K, tm, e, ma,
               mb, ma, mb, 0, none, e);
  }
  return launched();
}

namespace {
// Normal 128 x 256 tiles of one problem (N a multiple of 256) with the
// staged TMA-store epilogue where the output allows it.
bool group_maps(int M, int N, int K, const void* A, int lda, const void* W, int ldw, const EpiArgs& e, TileMap* tm,
                CUtensorMap* ma, CUtensorMap* mb, CUtensorMap* mo, CUtensorMap* mh) {
  *tm = {};
  tm->num_m = (M + BM - 1) / BM;
  tm->num_m2 = (M + 255) / 256;
  tm->n_full = N / 256;
  tm->n_norm = tm->num_m * tm->n_full;
  tm->n_tiles = tm->n_norm;
  if (!make_map(ma, A, M, K, lda, BM) || !make_map(mb, W, N, K, ldw, 256)) return false;
  *mo = *ma;
  *mh = *ma;
  const bool aligned = !((uintptr_t)e.out & 15) && e.ldo % 8 == 0 &&
                       (!e.hist_out || (!((uintptr_t)e.hist_out & 15) && !((uintptr_t)e.hist_base & 15)));
  const bool gate_ok = !e.gate || ((e.seg_split <= 0 || e.rpb0 >= 32) && e.rpb1 >= 32);
  if (!e.out_f32 && e.split_col >= N && aligned && gate_ok && make_store_map(mo, e.out, M, N, e.ldo) &&
      (!e.hist_out || make_store_map(mh, e.hist_out, M, N, e.ldo)))
    tm->staged = 1;
  return true;
}
}  // namespace

cudaError_t gemm_tc_grouped(int M0, const void* A0, const void* W0, const EpiArgs& e0, int M1, const void* A1,
                            const void* W1, const EpiArgs& e1, int N, int K, int lda, int ldw, cudaStream_t s) {
  if (M1 <= 0) return gemm_tc(M0, N, K, A0, lda, W0, ldw, e0, s);
  if (M0 <= 0) return gemm_tc(M1, N, K, A1, lda, W1, ldw, e1, s);
  if (!init_driver()) return cudaErrorNotSupported;
  if (!ln_ok(e0, N) || !ln_ok(e1, N) || (ln_side(e0) && ln_side(e1) && ln_side(e0) != ln_side(e1)))
    return cudaErrorInvalidValue;
  // long reductions: both problems in one CTA-pair launch (256-row tiles
  // of the image rows, then of the text rows)
  if (M0 >= 2 * BM && K >= 8192) {
    if (K % 8 != 0 || lda % 8 != 0 || ldw % 8 != 0 || N % 8 != 0) return cudaErrorInvalidValue;
    if (((uintptr_t)A0 & 15) || ((uintptr_t)W0 & 15) || ((uintptr_t)A1 & 15) || ((uintptr_t)W1 & 15))
      return cudaErrorInvalidValue;
    const int pairs = g_sms / 2;
    const long long rows_t = ((M0 + 2 * BM - 1) / (2 * BM)) + ((M1 + 2 * BM - 1) / (2 * BM));
    const int bn = pick_bn((int)(rows_t * 2 * BM), N, 2 * BM, pairs);
    CUtensorMap a0, b0, a1, b1;
    if (!make_map(&a0, A0, M0, K, lda, BM) || !make_map(&b0, W0, N, K, ldw, bn / 2) ||
        !make_map(&a1, A1, M1, K, lda, BM) || !make_map(&b1, W1, N, K, ldw, bn / 2))
      return cudaErrorInvalidValue;
    TileMap t0 = {}, t1 = {};
    CUtensorMap o0 = a0, h0 = a0, o1 = a1, h1 = a1;
    t0.staged = staged_maps(e0, M0, N, &o0, &h0) ? 1 : 0;
    t1.staged = staged_maps(e1, M1, N, &o1, &h1) ? 1 : 0;
    const long long tiles = rows_t * ((N + bn - 1) / bn);
    const int grid = 2 * (int)(tiles < pairs ? tiles : pairs);
    const int ln = std::max(ln_side(e0), ln_side(e1));
    if (bn == 256)
      launch_pdl(gemm2_fn<256, true>(ln), grid, THREADS, Cfg2<256>::SMEM, s, a0, b0, o0, h0, M0, N, K, t0, e0, a1, b1, o1,
                 h1, M1, t1, e1);
    else
      launch_pdl(gemm2_fn<128, true>(ln), grid, THREADS, Cfg2<128>::SMEM, s, a0, b0, o0, h0, M0, N, K, t0, e0, a1, b1, o1,
                 h1, M1, t1, e1);
    return launched();
  }
  // column counts that need swapped tiles run as two launches
  if (N % 256 != 0) {
    const cudaError_t r = gemm_tc(M1, N, K, A1, lda, W1, ldw, e1, s);
    return r != cudaSuccess ? r : gemm_tc(M0, N, K, A0, lda, W0, ldw, e0, s);
  }
  if (K % 8 != 0 || lda % 8 != 0 || ldw % 8 != 0) return cudaErrorInvalidValue;
  if (((uintptr_t)A0 & 15) || ((uintptr_t)W0 & 15) || ((uintptr_t)A1 & 15) || ((uintptr_t)W1 & 15))
    return cudaErrorInvalidValue;
  TileMap t0, t1;
  CUtensorMap a0, b0, o0, h0, a1, b1, o1, h1;
  if (!group_maps(M0, N, K, A0, lda, W0, ldw, e0, &t0, &a0, &b0, &o0, &h0) ||
      !group_maps(M1, N, K, A1, lda, W1, ldw, e1, &t1, &a1, &b1, &o1, &h1))
    return cudaErrorInvalidValue;
  const long long tiles = (long long)t0.n_tiles + t1.n_tiles;
  const int grid = (int)(tiles < g_sms ? tiles : g_sms);
  const int ln = std::max(ln_side(e0), ln_side(e1));
  launch_pdl(gemm_fn<256, true>(ln), grid, THREADS, Cfg<256>::SMEM, s, a0, b0, a0, a0, o0, h0, a0, a0, M0, N, K, t0, e0, a1,
             b1, o1, h1, M1, t1, e1);
  return launched();
}

// ---------------------------------------------------------------------------
// Watchdog probe (failure-detection test hook): one CTA takes TMEM like the
// GEMM does, then waits with the GEMM's bounded wait on an mbarrier that
// nothing arrives on.  The wait gives up after limit_ns, raises the same
// watchdog flag a stuck GEMM raises, and the CTA frees its TMEM and returns.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(64, 1) k_watchdog_probe(unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);   // one arrival expected; none comes
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(&tmem_slot)), "r"(32)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  if (lane == 0) mbar_wait<true>(&bar, 0, &abort_flag, &g_watchdog, limit_ns);
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(32) : "memory");
  }
}

cudaError_t watchdog_probe(unsigned long long limit_ns, cudaStream_t s) {
  k_watchdog_probe<<<1, 64, 0, s>>>(limit_ns);
  count_launches(1);
  return cudaGetLastError();
}

unsigned int gemm_tc_watchdog_take() {
  unsigned int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_watchdog, sizeof(v)) != cudaSuccess) return 0;
  if (v) cudaMemcpyToSymbol(g_watchdog, &z, sizeof(z));
  return v;
}

}  // namespace ff
