// Step A1, bf16 path -- non-causal GQA attention on the 5th-generation tensor
// cores (tcgen05, accumulators in tensor memory, operands staged by TMA).
//
// Sec. 4.2: the refiner corrects over the entire sequence, so every valid
// query attends to every valid key (no causal or block mask); Sec. 3.3 is the
// block-causal pattern it replaces. out = softmax(q k^T / sqrt(D)) v per
// (sequence, query head), kv head = floor(h * Hkv / Hq), varlen via seq_lens.
//
// Work unit: two 128-row query tiles that read the same key/value head of the
// same sequence (two query heads of one GQA group, or two row blocks of one
// head), so each 128-key K/V tile that TMA brings into shared memory feeds
// both. The kernel is persistent: one CTA per SM walks units
// blockIdx.x, blockIdx.x + gridDim.x, ... and overlaps the next unit's query
// load and first score MMAs with the current unit's last MMAs and epilogue.
//
// Warp roles (320 threads):
//   warps 0-3  softmax + epilogue of tile slot 0 (thread t owns query row t = TMEM lane t)
//   warps 4-7  softmax + epilogue of tile slot 1
//   warp 8     TMA producer (Q per unit and slot; K_0, V_0, K_1, V_1, ... through a
//              ring of four tile-sized slots, each released as soon as the MMAs
//              that read it have completed)
//   warp 9     tensor-memory allocator and MMA issuer (one elected thread)
// Tensor memory (512 columns x 128 lanes x 32 bit):
//   S_i = Q_i K_j^T  fp32, columns [128 i, 128 i + 128)
//   P_i = bf16 softmax numerators, written over the first 64 columns of S_i
//   O_i = sum_j P_i V_j fp32, columns [256 + D i, 256 + D i + D)
// MMA order per key tile j: PV_0(j), S_0(j+1), PV_1(j), S_1(j+1); after the
// last tile of a unit, S_0(0), S_1(0) of the next unit. The tensor pipe
// executes one thread's tcgen05.mma in issue order, so a score MMA overwrites
// P_i only after the PV MMA before it has read P_i.
// Online softmax in the log2 domain with exp2; the running maximum used for the
// numerators is raised (and O rescaled) only when it grows by more than 8,
// which bounds every numerator by 2^8 and leaves the final O / l exact.
//
// Barrier phases: every barrier completes once per event of one stream of
// events (per slot: query loads, score MMAs, numerator hand-offs, output
// hand-offs; per ring stage: fills and releases) and each waiter counts the
// events it has consumed, so parities line up across units without resets.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "dlm_common.cuh"
#include "dlm_internal.h"

namespace dlm {
namespace {

constexpr int kTile = 128;          // query rows per tile = keys per K/V tile
constexpr int kRing = 4;            // K/V ring: 32-KB slots holding K_c, V_c, K_c+1, ...
constexpr int kThreads = 320;
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp = 9;
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D>
struct Smem {
  static constexpr int kBoxBytes = kTile * 64 * 2;     // one 128 x 64 bf16 TMA box (16 KB)
  static constexpr int kTileBytes = kTile * D * 2;     // D / 64 boxes
  static constexpr int kStageBytes = 32 * 32 * 2;      // epilogue staging: 32 rows x 32 bf16
  alignas(1024) uint8_t q[2][kTileBytes];
  alignas(1024) uint8_t ring[kRing][kTileBytes];       // K_c, V_c, K_c+1, V_c+1, ...
  alignas(128) uint8_t stage[8][2][kStageBytes];       // per softmax warp, double-buffered
  uint64_t bar_q[2];          // query tile of slot i landed        (TMA -> MMA)
  uint64_t bar_qfree[2];      // last score MMA of slot i issued   (MMA -> TMA)
  uint64_t bar_full[kRing];   // ring slot filled (V padding cleared) (TMA -> MMA)
  uint64_t bar_empty[kRing];  // ring slot read by its MMAs         (MMA -> TMA)
  uint64_t bar_s[2];          // S_i ready                          (MMA -> softmax)
  uint64_t bar_p[2];          // P_i written, O_i rescaled          (softmax -> MMA)
  uint64_t bar_o[2];          // O_i final for the unit             (MMA -> epilogue)
  uint64_t bar_ofree[2];      // O_i read out by the epilogue       (epilogue -> MMA)
  uint64_t bar_vtmp;          // private fill of a partial V tile
  uint64_t bar_done;          // every MMA of this CTA completed
  uint32_t tmem_base;
  int abort;
};

struct TcParams {
  int B, L, Hq, Hkv, G, mtiles, units_per_bg, units;
  const int32_t* seq_lens;
  __nv_bfloat16* out;
  int64_t so0, so1, so2;
  float scale_log2;
  int* err;
};

struct Unit {
  int b, g, n, nkv;
  int head[2], row0[2];
  bool active[2], run[2];
};

__device__ __forceinline__ Unit decode_unit(const TcParams& p, int unit) {
  Unit U;
  const int bg = unit / p.units_per_bg;
  const int u = unit % p.units_per_bg;
  U.b = bg / p.Hkv;
  U.g = bg % p.Hkv;
  int n = p.seq_lens ? p.seq_lens[U.b] : p.L;
  if (n < 0 || n > p.L) {
    if (threadIdx.x == 0) set_device_error(p.err, DLM_DEVERR_LENGTH);
    n = n < 0 ? 0 : p.L;
  }
  U.n = n;
  const int ntiles = p.G * p.mtiles;
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int t = 2 * u + i;
    U.active[i] = t < ntiles;
    U.head[i] = U.g * p.G + (U.active[i] ? t % p.G : 0);
    U.row0[i] = (U.active[i] ? t / p.G : 0) * kTile;
    U.run[i] = U.active[i] && U.row0[i] < n;
  }
  U.nkv = (U.run[0] || U.run[1]) ? (n + kTile - 1) / kTile : 0;
  return U;
}

// Warp-uniform bounded wait: true only if every lane saw the phase complete.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort, int* err) {
  bool ok = mbar_wait(bar, parity, abort, err);
  return __all_sync(0xffffffffu, ok);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
                   const __grid_constant__ CUtensorMap tv, const __grid_constant__ CUtensorMap to,
                   const TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  Smem<D>& sm = *reinterpret_cast<Smem<D>*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  constexpr int kBoxes = D / 64;
  constexpr uint32_t kBoxBytes = Smem<D>::kBoxBytes;
  constexpr uint32_t kTileBytes = Smem<D>::kTileBytes;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // ---- setup (once per persistent CTA)
  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.bar_q[i], 1);
      mbar_init(&sm.bar_qfree[i], 1);
      mbar_init(&sm.bar_s[i], 1);
      mbar_init(&sm.bar_p[i], 128);
      mbar_init(&sm.bar_o[i], 1);
      mbar_init(&sm.bar_ofree[i], 128);
    }
    for (int r = 0; r < kRing; ++r) {
      mbar_init(&sm.bar_full[r], 1);
      mbar_init(&sm.bar_empty[r], 1);
    }
    mbar_init(&sm.bar_vtmp, 1);
    mbar_init(&sm.bar_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    fence_proxy_async_smem();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == kProducerWarp) {
    // ================================================================ TMA producer
    // Ring fills f = 0, 1, 2, ...: K_c at f = 2c, V_c at f = 2c + 1 (c counts the
    // key tiles of all units of this CTA); slot f % kRing, phase (f / kRing) & 1.
    int q_loads[2] = {0, 0};   // query loads per slot (= bar_q / bar_qfree phases)
    int fills = 0;             // ring fills issued
    int vtmp = 0;              // private partial-V fills
    bool ok = true;
    if (lane == 0) {
      prefetch_tmap(&tq);
      prefetch_tmap(&tk);
      prefetch_tmap(&tv);
      prefetch_tmap(&to);
    }
    auto acquire = [&](int f) -> bool {
      return f < kRing || warp_wait(&sm.bar_empty[f % kRing], ((f / kRing) - 1) & 1, abort, p.err);
    };
    for (int unit = blockIdx.x; ok && unit < p.units; unit += gridDim.x) {
      const Unit U = decode_unit(p, unit);
      if (U.nkv == 0) continue;
      for (int i = 0; i < 2 && ok; ++i) {
        if (!U.run[i]) continue;
        // The slot's previous query tile is free once its last score MMA has run.
        if (q_loads[i] > 0 && !warp_wait(&sm.bar_qfree[i], (q_loads[i] - 1) & 1, abort, p.err)) { ok = false; break; }
        if (lane == 0) {
          mbar_arrive_expect_tx(&sm.bar_q[i], kTileBytes);
          for (int c = 0; c < kBoxes; ++c)
            tma_load_4d(sm.q[i] + c * kBoxBytes, &tq, &sm.bar_q[i], 64 * c, U.head[i], U.row0[i], U.b);
        }
        ++q_loads[i];
      }
      for (int j = 0; ok && j < U.nkv; ++j) {
        // K_j
        if (!acquire(fills)) { ok = false; break; }
        {
          const int r = fills % kRing;
          if (lane == 0) {
            mbar_arrive_expect_tx(&sm.bar_full[r], kTileBytes);
            for (int c = 0; c < kBoxes; ++c)
              tma_load_4d(sm.ring[r] + c * kBoxBytes, &tk, &sm.bar_full[r], 64 * c, U.g, j * kTile, U.b);
          }
          ++fills;
        }
        // V_j
        if (!acquire(fills)) { ok = false; break; }
        const int r = fills % kRing;
        const int valid = U.n - j * kTile;
        if (valid >= kTile) {
          if (lane == 0) {
            mbar_arrive_expect_tx(&sm.bar_full[r], kTileBytes);
            for (int c = 0; c < kBoxes; ++c)
              tma_load_4d(sm.ring[r] + c * kBoxBytes, &tv, &sm.bar_full[r], 64 * c, U.g, j * kTile, U.b);
          }
          ++fills;
        } else {
          // Last, partial tile: value rows >= n may hold any bit pattern and a
          // zero softmax weight does not cancel a NaN/Inf, so clear them in
          // shared memory before the MMA reads the tile.
          if (lane == 0) {
            mbar_arrive_expect_tx(&sm.bar_vtmp, kTileBytes);
            for (int c = 0; c < kBoxes; ++c)
              tma_load_4d(sm.ring[r] + c * kBoxBytes, &tv, &sm.bar_vtmp, 64 * c, U.g, j * kTile, U.b);
          }
          ++vtmp;
          if (!warp_wait(&sm.bar_vtmp, (vtmp - 1) & 1, abort, p.err)) { ok = false; break; }
          const int zrows = kTile - valid;
          for (int c = 0; c < kBoxes; ++c) {
            uint4* base = reinterpret_cast<uint4*>(sm.ring[r] + c * kBoxBytes + valid * 128);
            for (int e = lane; e < zrows * 8; e += 32) base[e] = make_uint4(0u, 0u, 0u, 0u);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.bar_full[r]);
          ++fills;
        }
      }
    }
    // Teardown: let every copy this warp issued land before the block exits.
    if (lane == 0) {
      for (int i = 0; i < 2; ++i)
        if (q_loads[i]) mbar_drain(&sm.bar_q[i], (q_loads[i] - 1) & 1);
      if (vtmp) mbar_drain(&sm.bar_vtmp, (vtmp - 1) & 1);
      for (int r = 0; r < kRing; ++r) {
        const int n_r = fills > r ? (fills - r + kRing - 1) / kRing : 0;  // fills of slot r
        if (n_r) mbar_drain(&sm.bar_full[r], (n_r - 1) & 1);
      }
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ================================================================ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(128, 128, false, false);  // Q, K both K-major
      constexpr uint32_t idesc_o = idesc_bf16_f32(128, D, false, true);     // V is MN-major (D contiguous)
      const uint32_t q_addr[2] = {smem_u32(sm.q[0]), smem_u32(sm.q[1])};
      auto issue_s = [&](int i, int r) {
        const uint32_t kaddr = smem_u32(sm.ring[r]);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk / 4) * kBoxBytes + (kk % 4) * 32;
          mma_ss(tmem + 128 * i, sdesc_sw128(q_addr[i] + off, 16, 1024), sdesc_sw128(kaddr + off, 16, 1024),
                 idesc_s, kk > 0);
        }
        mma_commit(&sm.bar_s[i]);
      };
      auto issue_pv = [&](int i, int r, bool acc) {
        const uint32_t vaddr = smem_u32(sm.ring[r]);
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          mma_ts(tmem + 256 + D * i, tmem + 128 * i + kk * 8, sdesc_sw128(vaddr + kk * 16 * 128, kBoxBytes, 1024),
                 idesc_o, (acc || kk > 0) ? 1u : 0u);
        }
      };
      auto wait_fill = [&](int f) -> bool {
        return mbar_wait(&sm.bar_full[f % kRing], (f / kRing) & 1, abort, p.err);
      };
      int q_loads[2] = {0, 0};   // bar_q phases consumed per slot
      int units_run[2] = {0, 0}; // bar_o / bar_ofree phases per slot
      int p_seen[2] = {0, 0};    // bar_p phases consumed per slot
      int tiles = 0;             // key tiles consumed (ring fill of K_c is 2c, of V_c is 2c + 1)
      bool ok = true;
      for (int unit = blockIdx.x; ok && unit < p.units; unit += gridDim.x) {
        const Unit U = decode_unit(p, unit);
        if (U.nkv == 0) continue;
        const int last_slot = U.run[1] ? 1 : 0;
        for (int i = 0; i < 2 && ok; ++i) {
          if (!U.run[i]) continue;
          ok = mbar_wait(&sm.bar_q[i], q_loads[i] & 1, abort, p.err);
          ++q_loads[i];
        }
        if (!ok || !wait_fill(2 * tiles)) break;
        tc_fence_after();
        for (int i = 0; i < 2; ++i) {
          if (!U.run[i]) continue;
          issue_s(i, (2 * tiles) % kRing);
          if (U.nkv == 1) mma_commit(&sm.bar_qfree[i]);
        }
        mma_commit(&sm.bar_empty[(2 * tiles) % kRing]);
        for (int j = 0; ok && j < U.nkv; ++j) {
          const int c = tiles + j;
          const int fv = 2 * c + 1, fk = 2 * c + 2;
          const bool next = j + 1 < U.nkv;
          if (!wait_fill(fv)) { ok = false; break; }
          bool k_ready = false;
          for (int i = 0; i < 2 && ok; ++i) {
            if (!U.run[i]) continue;
            // O_i of this slot's previous unit must have been read out before PV(0) overwrites it.
            if (j == 0 && units_run[i] > 0 &&
                !mbar_wait(&sm.bar_ofree[i], (units_run[i] - 1) & 1, abort, p.err)) {
              ok = false;
              break;
            }
            if (!mbar_wait(&sm.bar_p[i], p_seen[i] & 1, abort, p.err)) { ok = false; break; }
            ++p_seen[i];
            tc_fence_after();
            issue_pv(i, fv % kRing, j > 0);
            if (!next) mma_commit(&sm.bar_o[i]);
            if (i == last_slot) mma_commit(&sm.bar_empty[fv % kRing]);
            if (next) {
              if (!k_ready) {
                if (!wait_fill(fk)) { ok = false; break; }
                tc_fence_after();
                k_ready = true;
              }
              issue_s(i, fk % kRing);
              if (j + 2 == U.nkv) mma_commit(&sm.bar_qfree[i]);
              if (i == last_slot) mma_commit(&sm.bar_empty[fk % kRing]);
            }
          }
        }
        tiles += U.nkv;
        for (int i = 0; i < 2; ++i)
          if (U.run[i]) ++units_run[i];
      }
      // Teardown: every MMA issued by this thread completes before TMEM is freed.
      mma_commit(&sm.bar_done);
      mbar_drain(&sm.bar_done, 0);
    }
    __syncwarp();
  } else {
    // ================================================================ softmax + epilogue
    const int i = warp >> 2;                 // tile slot
    const int qw = warp & 3;                 // warp within the warpgroup: rows 32 qw .. 32 qw + 31
    const int t = threadIdx.x & 127;         // row within the tile = TMEM lane
    const uint32_t lane_base = static_cast<uint32_t>(qw * 32) << 16;
    const uint32_t s_addr = tmem + lane_base + 128 * i;
    const uint32_t o_addr = tmem + lane_base + 256 + D * i;
    int s_seen = 0;     // bar_s phases consumed
    int units_run = 0;  // bar_o phases consumed
    bool ok = true;
    for (int unit = blockIdx.x; ok && unit < p.units; unit += gridDim.x) {
      const Unit U = decode_unit(p, unit);
      if (!U.active[i]) continue;
      const int row = U.row0[i] + t;
      if (!U.run[i]) {
        // Every row of this tile is padding: zeros.
        if (row < p.L) {
          uint4* dst = reinterpret_cast<uint4*>(p.out + U.b * p.so0 + static_cast<int64_t>(row) * p.so1 +
                                                U.head[i] * p.so2);
#pragma unroll
          for (int e = 0; e < D / 8; ++e) dst[e] = make_uint4(0u, 0u, 0u, 0u);
        }
        continue;
      }
      float m_used = -INFINITY;
      float l = 0.f;
      for (int j = 0; j < U.nkv; ++j) {
        if (!warp_wait(&sm.bar_s[i], s_seen & 1, abort, p.err)) { ok = false; break; }
        ++s_seen;
        tc_fence_after();
        uint32_t sr[128];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(s_addr + 32 * c, *reinterpret_cast<uint32_t(*)[32]>(&sr[32 * c]));
        tmem_wait_ld();
        float sv[128];
#pragma unroll
        for (int c = 0; c < 128; ++c) sv[c] = __uint_as_float(sr[c]);
        const int valid = U.n - j * kTile;
        if (valid < kTile) {
#pragma unroll
          for (int c = 0; c < 128; ++c)
            if (c >= valid) sv[c] = -INFINITY;
        }
        float mx0 = sv[0], mx1 = sv[1], mx2 = sv[2], mx3 = sv[3];
#pragma unroll
        for (int c = 4; c < 128; c += 4) {
          mx0 = fmaxf(mx0, sv[c]);
          mx1 = fmaxf(mx1, sv[c + 1]);
          mx2 = fmaxf(mx2, sv[c + 2]);
          mx3 = fmaxf(mx3, sv[c + 3]);
        }
        const float m_tile = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * p.scale_log2;
        const bool raise = m_tile > m_used + kRescaleThreshold;
        if (__any_sync(0xffffffffu, raise)) {
          const float m_new = raise ? m_tile : m_used;
          const float alpha = (m_used == -INFINITY) ? 0.f : ex2_approx(m_used - m_new);
          l *= alpha;
          m_used = m_new;
          if (j > 0) {
            // O holds sum_{j' < j} P V (the score MMA of tile j was issued after
            // the PV MMA of tile j-1, and bar_s has completed): rescale it.
#pragma unroll 1
            for (int c = 0; c < D / 32; ++c) {
              uint32_t ov[32];
              tmem_ld32(o_addr + 32 * c, ov);
              tmem_wait_ld();
#pragma unroll
              for (int e = 0; e < 32; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * alpha);
              tmem_st32(o_addr + 32 * c, ov);
            }
          }
        }
        uint32_t pk[64];
        float l0 = 0.f, l1 = 0.f;
#pragma unroll
        for (int c = 0; c < 64; ++c) {
          const float p0 = ex2_approx(fmaf(sv[2 * c], p.scale_log2, -m_used));
          const float p1 = ex2_approx(fmaf(sv[2 * c + 1], p.scale_log2, -m_used));
          l0 += p0;
          l1 += p1;
          pk[c] = pack_bf16x2(p0, p1);
        }
        l += l0 + l1;
        tmem_st32(s_addr, *reinterpret_cast<const uint32_t(*)[32]>(&pk[0]));
        tmem_st32(s_addr + 32, *reinterpret_cast<const uint32_t(*)[32]>(&pk[32]));
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(&sm.bar_p[i]);
      }
      if (!ok || !warp_wait(&sm.bar_o[i], units_run & 1, abort, p.err)) { ok = false; break; }
      ++units_run;
      // Epilogue: read O_i out of tensor memory, hand the columns back to the
      // MMA warp, then normalise, convert to bf16, stage 32 rows x 32 columns
      // per warp in shared memory and write them with TMA stores (rows >= n
      // are zero; rows >= L are clipped by the tensor map).
      tc_fence_after();
      uint32_t ov[D];
#pragma unroll
      for (int c = 0; c < D / 32; ++c) tmem_ld32(o_addr + 32 * c, *reinterpret_cast<uint32_t(*)[32]>(&ov[32 * c]));
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(&sm.bar_ofree[i]);
      const bool valid_row = row < U.n;
      const float inv = valid_row ? 1.0f / l : 0.f;
      const int wrow0 = U.row0[i] + 32 * qw;
      if (wrow0 < p.L) {
        if (lane == 0) bulk_wait_read<0>();  // staging buffers of the previous unit are free
        __syncwarp();
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint8_t* buf = sm.stage[warp][c & 1];
          if (c >= 2) {
            if (lane == 0) bulk_wait_read<1>();
            __syncwarp();
          }
          uint4* dst = reinterpret_cast<uint4*>(buf + lane * 64);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            uint32_t w[4];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const int col = 32 * c + 8 * e + 2 * h;
              w[h] = valid_row ? pack_bf16x2(__uint_as_float(ov[col]) * inv, __uint_as_float(ov[col + 1]) * inv)
                               : 0u;
            }
            dst[e] = make_uint4(w[0], w[1], w[2], w[3]);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_4d(&to, buf, 32 * c, U.head[i], wrow0, U.b);
            bulk_commit();
          }
        }
      }
    }
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------- host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// 4-D map over a [B, L, H, D] bf16 tensor with element strides (sb, sl, sh, 1);
// box = box_d head-dim elements x 1 head x box_rows rows x 1 sequence.
int make_map(CUtensorMap* map, const void* base, int B, int L, int H, int D, const int64_t* s, int box_d = 64,
             int box_rows = kTile, CUtensorMapSwizzle swz = CU_TENSOR_MAP_SWIZZLE_128B) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return fail(DLM_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(H), static_cast<cuuint64_t>(L),
                        static_cast<cuuint64_t>(B)};
  cuuint64_t strides[3] = {static_cast<cuuint64_t>(s[2]) * 2, static_cast<cuuint64_t>(s[1]) * 2,
                           static_cast<cuuint64_t>(s[0]) * 2};
  cuuint32_t box[4] = {static_cast<cuuint32_t>(box_d), 1, static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(DLM_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return DLM_OK;
}

template <int D>
int launch_d(const AttnArgs& a, cudaStream_t stream) {
  CUtensorMap mq, mk, mv, mo;
  int st;
  if ((st = make_map(&mq, a.q, a.B, a.L, a.Hq, D, a.sq)) != DLM_OK) return st;
  if ((st = make_map(&mk, a.k, a.B, a.L, a.Hkv, D, a.sk)) != DLM_OK) return st;
  if ((st = make_map(&mv, a.v, a.B, a.L, a.Hkv, D, a.sv)) != DLM_OK) return st;
  // Output: 32 x 32 boxes (one warp's rows, one 64-byte column chunk), no swizzle.
  if ((st = make_map(&mo, a.out, a.B, a.L, a.Hq, D, a.so, 32, 32, CU_TENSOR_MAP_SWIZZLE_NONE)) != DLM_OK) return st;
  TcParams p;
  p.B = a.B;
  p.L = a.L;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.G = a.Hq / a.Hkv;
  p.mtiles = (a.L + kTile - 1) / kTile;
  p.units_per_bg = (p.G * p.mtiles + 1) / 2;
  const long long units = static_cast<long long>(a.B) * a.Hkv * p.units_per_bg;
  if (units == 0) return DLM_OK;
  if (units > 0x7FFFFFFFLL) return fail(DLM_ERR_SHAPE, "too many attention work units");
  p.units = static_cast<int>(units);
  p.seq_lens = a.seq_lens;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.so0 = a.so[0];
  p.so1 = a.so[1];
  p.so2 = a.so[2];
  p.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(D));
  p.err = device_error_word();
  const size_t smem = sizeof(Smem<D>) + 1024;
  cudaError_t attr_err = cudaFuncSetAttribute(attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              static_cast<int>(smem));
  if (attr_err != cudaSuccess) return fail(DLM_ERR_CUDA, "attn smem attribute: %s", cudaGetErrorString(attr_err));
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = static_cast<int>(units < sms ? units : sms);
  attn_tc_kernel<D><<<grid, kThreads, smem, stream>>>(mq, mk, mv, mo, p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "attn_tc launch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

}  // namespace

int launch_attn_tc_bf16(const AttnArgs& a, cudaStream_t stream) {
  if (a.B == 0 || a.L == 0) return DLM_OK;
  return a.D == 64 ? launch_d<64>(a, stream) : launch_d<128>(a, stream);
}

}  // namespace dlm
