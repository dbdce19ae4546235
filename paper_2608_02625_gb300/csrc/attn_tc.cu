// Step A1, bf16 path -- non-causal GQA attention on the 5th-generation tensor
// cores (tcgen05, accumulators in tensor memory, operands staged by TMA).
//
// Sec. 4.2: the refiner corrects over the entire sequence, so every valid
// query attends to every valid key (no causal or block mask); Sec. 3.3 is the
// block-causal pattern it replaces. out = softmax(q k^T / sqrt(D)) v per
// (sequence, query head), kv head = floor(h * Hkv / Hq), varlen via seq_lens.
//
// Work unit: two 128-row query tiles ("slots") that read the same key/value
// head of the same sequence (two query heads of one GQA group, or two row
// blocks of one head), so each key/value tile staged in shared memory feeds
// both. When even single tiles all fit on the SMs at once (a single short
// sequence) a unit is one tile in slot 0 and slot 1 idles. The kernel
// is persistent: one CTA per SM walks units blockIdx.x, blockIdx.x +
// gridDim.x, ...; the next unit's query tiles load as soon as the slot's last
// score MMA has run, and its first score MMAs overlap the epilogue.
//
// Keys are processed in 64-key sub-tiles so that each slot's scores can be
// double-buffered in tensor memory: the tensor core computes S(j+1) while the
// softmax warps work on S(j), which keeps the serial chain
// softmax -> PV -> next scores off the critical path.
//
// Warp roles (352 threads):
//   warps 0-3  softmax + epilogue of slot 0 (thread t owns query row t = TMEM lane t)
//   warps 4-7  softmax + epilogue of slot 1
//   warp 8     TMA producer: Q per unit and slot; then the unit's key/value
//              sub-tiles through a ring of four entries of two sub-tiles each,
//              in the order the issuers consume them -- [K_0 | K_1], then
//              [V_j | K_{j+2}] for each j -- so that each step of an issuer
//              waits for one fill; an entry is released, per slot, by the
//              slot's softmax warps once they see the completion of the MMAs
//              that read it (no tcgen05.commit for it in the issuer)
//   warp 9     tensor-memory allocator; MMA issuer of slot 0 (one lane elected
//              per instruction)
//   warp 10    MMA issuer of slot 1
// Tensor memory (512 columns x 128 lanes x 32 bit), slot i at column 256 i:
//   S_i buffers 0 and 1   fp32 128 x 64 at +0 and +64 (sub-tile j uses buffer j % 2)
//   P_i                    bf16 numerators over the first 32 columns of that buffer
//   O_i = sum_j P_i V_j    fp32 128 x D at +128
// MMA order of slot i per sub-tile j: PV_i(j), S_i(j+2). The tensor pipe
// executes one thread's tcgen05.mma in issue order, so S(j+2) overwrites the
// buffer holding P(j) only after PV(j) has read it. Each slot has its own
// issuing thread: issue blocks while the tensor pipe's queue is full, so one
// thread alone would leave the pipe idle during each of its waits. At the
// start of every unit slot 1's softmax waits for slot 0's first hand-off, so
// the two slots run half a step apart and their MMA bursts alternate with
// the other slot's softmax instead of coinciding.
// Online softmax in the log2 domain with exp2; the running maximum used for the
// numerators is raised (and O rescaled, after the previous PV has completed)
// only when it grows by more than 8, which bounds every numerator by 2^8 and
// leaves the final O / l exact.
//
// Barrier phases: each barrier completes once per event of one ordered stream
// (per slot: query loads, score MMAs per buffer, numerator hand-offs, PV
// completions, output hand-offs; per ring slot: fills and releases) and every
// waiter counts the events it consumed. Each wait is arranged so that the
// barrier cannot run two phases ahead of its waiter (the next event needs
// something the waiter only provides after the wait), so parities never alias.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "dlm_common.cuh"
#include "dlm_internal.h"

namespace dlm {
namespace {

constexpr int kTile = 128;          // query rows per tile
constexpr int kSub = 64;            // keys per sub-tile
constexpr int kRing = 4;            // K/V ring entries (two sub-tiles each)
constexpr int kThreads = 352;
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp0 = 9;   // warps 9 and 10 issue the MMAs of slots 0 and 1
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D>
struct Smem {
  static constexpr int kQBoxBytes = kTile * 64 * 2;    // Q box: 128 rows x 64 bf16 (16 KB)
  static constexpr int kQBytes = kTile * D * 2;        // D / 64 boxes
  static constexpr int kKvBoxBytes = kSub * 64 * 2;    // K/V box: 64 rows x 64 bf16 (8 KB)
  static constexpr int kKvBytes = kSub * D * 2;
  static constexpr int kStageBytes = 32 * 32 * 2;      // epilogue staging: 32 rows x 32 bf16
  alignas(1024) uint8_t q[2][kQBytes];
  alignas(1024) uint8_t ring[kRing][2][kKvBytes];      // [K_0 | K_1], [V_0 | K_2], [V_1 | K_3], ...
  alignas(1024) uint8_t stage[8][2][kStageBytes];       // per softmax warp, double-buffered
  uint64_t bar_q[2];          // query tile of slot i landed          (TMA -> MMA)
  uint64_t bar_qfree[2];      // last score MMA of slot i completed   (MMA -> TMA)
  uint64_t bar_full[kRing];   // ring slot filled (V padding cleared)  (TMA -> MMA)
  uint64_t bar_empty[kRing];  // ring slot read by its MMAs, per slot (softmax or idle issuer -> TMA)
  uint64_t bar_s[2][2];       // S_i buffer b ready                   (MMA -> softmax)
  uint64_t bar_p[2][2];       // hand-off n of slot i (P written, O rescaled) on bar_p[i][n % 2] (softmax -> MMA)
  uint64_t bar_pvm[2];        // the unit's next-to-last PV of slot i completed (MMA -> softmax)
  uint64_t bar_o[2];          // the unit's last PV of slot i completed: O_i final (MMA -> epilogue)
  uint64_t bar_ofree[2];      // O_i read out by the epilogue         (epilogue -> MMA)
  uint64_t bar_vtmp;          // private fill of a partial V sub-tile
  uint64_t bar_done[2];       // every MMA of issuer i completed
  uint32_t tmem_base;
  int abort;
  int unit_flag;   // units whose first slot-0 hand-off happened
};

// Division by a divisor fixed at launch as a multiply-high and a shift
// (Granlund and Montgomery, "Division by invariant integers using
// multiplication", PLDI 1994): for 0 <= n < 2^31 and d >= 1, with
// l = ceil(log2 d) and m = floor(2^(32 + l) / d) - 2^32 + 1,
// n / d = (umulhi(n, m) + n) >> l (the sum stays below 2^32).
struct FastDiv {
  uint32_t d, m, l;
  __device__ __forceinline__ int div(int n) const {
    const uint32_t u = static_cast<uint32_t>(n);
    return static_cast<int>((__umulhi(u, m) + u) >> l);
  }
};

FastDiv make_fastdiv(int d) {
  FastDiv f;
  f.d = static_cast<uint32_t>(d);
  f.l = 0;
  while ((1ull << f.l) < f.d) ++f.l;
  f.m = static_cast<uint32_t>((1ull << (32 + f.l)) / f.d - (1ull << 32) + 1);
  return f;
}

struct TcParams {
  int B, L, Hq, Hkv, G, mtiles, units_per_bg, units;
  int tpu;  // query tiles per unit: 2 (both slots), 1 (slot 0 only: few tiles)
  FastDiv div_upb, div_hkv, div_g;  // by units_per_bg, Hkv, G
  int mask_mode, block;
  const int32_t* seq_lens;
  const int32_t* prompt_lens;
  __nv_bfloat16* out;
  int64_t so0, so1, so2;
  float scale_log2;
  int* err;
  uint64_t wait_ns;  // budget of each bounded wait
};

// A value per slot, read with a select: the slot index comes from the warp,
// and an array indexed by it would live in local memory.
struct Pair {
  int v0, v1;
  __device__ __forceinline__ int operator[](int i) const { return i ? v1 : v0; }
};

struct Unit {
  int b, g, n, p, nkv;  // nkv: 64-key sub-tiles visited
  int ka, kgap;         // sub-tile j of the unit is key sub-tile kt(j) = j < ka ? j : j + kgap
  Pair head, row0, active, run;
  __device__ __forceinline__ int kt(int j) const { return j < ka ? j : j + kgap; }
};

template <bool kMasked>
__device__ __forceinline__ Unit decode_unit(const TcParams& p, int unit) {
  Unit U;
  const int bg = p.div_upb.div(unit);
  const int u = unit - bg * p.units_per_bg;
  U.b = p.div_hkv.div(bg);
  U.g = bg - U.b * p.Hkv;
  int n = p.seq_lens ? p.seq_lens[U.b] : p.L;
  if (n < 0 || n > p.L) {
    if (threadIdx.x == 0) set_device_error(p.err, DLM_DEVERR_LENGTH);
    n = n < 0 ? 0 : p.L;
  }
  U.n = n;
  const int ntiles = p.G * p.mtiles;
  {
    const int t0 = p.tpu * u, t1 = p.tpu == 2 ? t0 + 1 : ntiles;
    U.active.v0 = t0 < ntiles;
    U.active.v1 = t1 < ntiles;
    const int r0 = p.div_g.div(t0), r1 = p.div_g.div(t1);
    U.head.v0 = U.g * p.G + (U.active.v0 ? t0 - r0 * p.G : 0);
    U.head.v1 = U.g * p.G + (U.active.v1 ? t1 - r1 * p.G : 0);
    U.row0.v0 = (U.active.v0 ? r0 : 0) * kTile;
    U.row0.v1 = (U.active.v1 ? r1 : 0) * kTile;
    U.run.v0 = U.active.v0 && U.row0.v0 < n;
    U.run.v1 = U.active.v1 && U.row0.v1 < n;
  }
  U.p = 0;
  U.ka = U.nkv = (U.run[0] || U.run[1]) ? (n + kSub - 1) / kSub : 0;
  U.kgap = 0;
  if (kMasked && U.nkv > 0) {
    int pl = p.prompt_lens ? p.prompt_lens[U.b] : 0;
    if (pl < 0 || pl > n) {
      if (threadIdx.x == 0) set_device_error(p.err, DLM_DEVERR_LENGTH);
      pl = pl < 0 ? 0 : n;
    }
    U.p = pl;
    // Key sub-tiles any running row of the unit may use: [0, p) and the span
    // of the rows' blocks (ranges are monotone in the row).
    int r_lo = n, r_hi = -1;
    for (int i = 0; i < 2; ++i) {
      if (!U.run[i]) continue;
      r_lo = min(r_lo, U.row0[i]);
      r_hi = max(r_hi, min(U.row0[i] + kTile, n) - 1);
    }
    const KeyRanges lo = key_ranges(p.mask_mode, p.block, r_lo, n, pl);
    const KeyRanges hi = key_ranges(p.mask_mode, p.block, r_hi, n, pl);
    if (p.mask_mode == DLM_ATTN_BLOCK_CAUSAL || r_hi < pl) {
      U.ka = U.nkv = (hi.hi1 + kSub - 1) / kSub;
    } else {
      const int a_end = (pl + kSub - 1) / kSub;              // prompt sub-tiles
      const int c0 = (r_lo < pl ? pl : lo.lo2) / kSub;         // first sub-tile of the lowest block
      const int c1 = (hi.hi2 + kSub - 1) / kSub;
      if (c0 <= a_end) {
        U.ka = U.nkv = max(a_end, c1);
      } else {
        U.ka = a_end;
        U.kgap = c0 - a_end;
        U.nkv = a_end + (c1 - c0);
      }
    }
  }
  return U;
}

// Ring entries of a unit with nkv sub-tiles: [K_0 | K_1] (K_1 when nkv > 1),
// then for each j the entry [V_j | K_{j+2}] (K_{j+2} when it exists), which
// holds the two tiles one step of an issuer reads: PV(j) and S(j + 2). The
// producer and the MMA issuers walk the same order.

// Bits [a - key0, b - key0) of a 64-bit word, clamped to [0, 64): the keys
// a <= key < b of the sub-tile that starts at key0.
__device__ __forceinline__ uint64_t key_bits(int key0, int a, int b) {
  const int lo = max(a - key0, 0), hi = min(b - key0, 64);
  if (hi <= lo) return 0ull;
  const uint64_t below_hi = hi >= 64 ? ~0ull : (1ull << hi) - 1ull;
  return below_hi & ~((1ull << lo) - 1ull);  // lo < hi <= 64
}

// Warp-uniform bounded wait: true only if every lane saw the phase complete.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort, int* err,
                                          uint64_t budget_ns) {
  bool ok = mbar_wait_for(bar, parity, abort, err, budget_ns);
  return __all_sync(0xffffffffu, ok);
}

// kMasked: the block masks of dlm_attn_masked (a separate instantiation, so
// that full attention carries none of their per-row bookkeeping).
template <int D, bool kMasked>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
                   const __grid_constant__ CUtensorMap tv, const __grid_constant__ CUtensorMap to,
                   const TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  Smem<D>& sm = *reinterpret_cast<Smem<D>*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  constexpr int kBoxes = D / 64;
  constexpr uint32_t kQBoxBytes = Smem<D>::kQBoxBytes;
  constexpr uint32_t kQBytes = Smem<D>::kQBytes;
  constexpr uint32_t kKvBoxBytes = Smem<D>::kKvBoxBytes;
  constexpr uint32_t kKvBytes = Smem<D>::kKvBytes;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // ---- setup (once per persistent CTA)
  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.bar_q[i], 1);
      mbar_init(&sm.bar_qfree[i], 1);
      mbar_init(&sm.bar_s[i][0], 1);
      mbar_init(&sm.bar_s[i][1], 1);
      mbar_init(&sm.bar_p[i][0], 128);
      mbar_init(&sm.bar_p[i][1], 128);
      mbar_init(&sm.bar_pvm[i], 1);
      mbar_init(&sm.bar_o[i], 1);
      mbar_init(&sm.bar_ofree[i], 128);
    }
    for (int r = 0; r < kRing; ++r) {
      mbar_init(&sm.bar_full[r], 1);
      mbar_init(&sm.bar_empty[r], 2);  // one release per slot
    }
    mbar_init(&sm.bar_vtmp, 1);
    mbar_init(&sm.bar_done[0], 1);
    mbar_init(&sm.bar_done[1], 1);
    sm.abort = 0;
    sm.unit_flag = 0;
    fence_mbar_init();
    fence_proxy_async_smem();
  }
  if (warp == kMmaWarp0) {
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
    int q_loads0 = 0, q_loads1 = 0;  // query loads per slot (= bar_q / bar_qfree phases)
    int fills = 0;             // ring fills issued; slot fills % kRing, phase (fills / kRing) & 1
    int vtmp = 0;              // private partial-V fills
    bool ok = true;
    if (lane == 0) {
      prefetch_tmap(&tq);
      prefetch_tmap(&tk);
      prefetch_tmap(&tv);
      prefetch_tmap(&to);
    }
    // Loads one ring entry: part 0 = K_ja (prologue) or V_ja, part 1 = K_jb
    // (jb < 0: none), completing bar_full of the entry once.
    auto load_kv = [&](uint8_t* dst, const CUtensorMap* m, uint64_t* bar, int key0, const Unit& U) {
      for (int c = 0; c < kBoxes; ++c) tma_load_4d(dst + c * kKvBoxBytes, m, bar, 64 * c, U.g, key0, U.b);
    };
    auto fill = [&](const Unit& U, int ja, bool a_is_v, int jb) -> bool {
      const int r = fills % kRing;
      if (fills >= kRing && !warp_wait(&sm.bar_empty[r], ((fills / kRing) - 1) & 1, abort, p.err, p.wait_ns)) return false;
      const int key_a = (kMasked ? U.kt(ja) : ja) * kSub;
      const int key_b = jb >= 0 ? (kMasked ? U.kt(jb) : jb) * kSub : 0;
      const uint32_t b_bytes = jb >= 0 ? kKvBytes : 0u;
      const int valid = U.n - key_a;
      if (!a_is_v || valid >= kSub) {
        if (lane == 0) {
          mbar_arrive_expect_tx(&sm.bar_full[r], kKvBytes + b_bytes);
          load_kv(sm.ring[r][0], a_is_v ? &tv : &tk, &sm.bar_full[r], key_a, U);
          if (jb >= 0) load_kv(sm.ring[r][1], &tk, &sm.bar_full[r], key_b, U);
        }
      } else {
        // Last, partial value sub-tile: rows >= n may hold any bit pattern and
        // a zero softmax weight does not cancel a NaN/Inf, so clear them in
        // shared memory before the MMA reads the tile.
        if (lane == 0) {
          mbar_arrive_expect_tx(&sm.bar_vtmp, kKvBytes);
          load_kv(sm.ring[r][0], &tv, &sm.bar_vtmp, key_a, U);
        }
        ++vtmp;
        if (!warp_wait(&sm.bar_vtmp, (vtmp - 1) & 1, abort, p.err, p.wait_ns)) return false;
        const int zrows = kSub - valid;
        for (int c = 0; c < kBoxes; ++c) {
          uint4* base = reinterpret_cast<uint4*>(sm.ring[r][0] + c * kKvBoxBytes + valid * 128);
          for (int e = lane; e < zrows * 8; e += 32) base[e] = make_uint4(0u, 0u, 0u, 0u);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          if (jb >= 0) {
            mbar_arrive_expect_tx(&sm.bar_full[r], b_bytes);
            load_kv(sm.ring[r][1], &tk, &sm.bar_full[r], key_b, U);
          } else {
            mbar_arrive(&sm.bar_full[r]);
          }
        }
      }
      ++fills;
      return true;
    };
    for (int unit = blockIdx.x; ok && unit < p.units; unit += gridDim.x) {
      const Unit U = decode_unit<kMasked>(p, unit);
      if (U.nkv == 0) continue;
      // The unit's first key tiles need only ring slots: start them before
      // the query tiles, which wait for the previous unit's last score MMAs.
      ok = fill(U, 0, false, U.nkv >= 2 ? 1 : -1);
      for (int i = 0; i < 2 && ok; ++i) {
        if (!U.run[i]) continue;
        // The slot's previous query tile is free once its last score MMA has run.
        const int ql = i ? q_loads1 : q_loads0;
        if (ql > 0 && !warp_wait(&sm.bar_qfree[i], (ql - 1) & 1, abort, p.err, p.wait_ns)) { ok = false; break; }
        if (lane == 0) {
          mbar_arrive_expect_tx(&sm.bar_q[i], kQBytes);
          for (int c = 0; c < kBoxes; ++c)
            tma_load_4d(sm.q[i] + c * kQBoxBytes, &tq, &sm.bar_q[i], 64 * c, U.head[i], U.row0[i], U.b);
        }
        if (i) ++q_loads1; else ++q_loads0;
      }
      if (!ok) break;
      for (int j = 0; ok && j < U.nkv; ++j) ok = fill(U, j, true, j + 2 < U.nkv ? j + 2 : -1);
    }
    // Teardown: let every copy this warp issued land before the block exits.
    if (lane == 0) {
      if (q_loads0) mbar_drain(&sm.bar_q[0], (q_loads0 - 1) & 1);
      if (q_loads1) mbar_drain(&sm.bar_q[1], (q_loads1 - 1) & 1);
      if (vtmp) mbar_drain(&sm.bar_vtmp, (vtmp - 1) & 1);
      for (int r = 0; r < kRing; ++r) {
        const int n_r = fills > r ? (fills - r + kRing - 1) / kRing : 0;  // fills of slot r
        if (n_r) mbar_drain(&sm.bar_full[r], (n_r - 1) & 1);
      }
    }
    __syncwarp();
  } else if (warp >= kMmaWarp0) {
    // ================================================================ MMA issuers
    // Warp kMmaWarp0 + i issues every MMA of slot i, so the two slots' MMA
    // streams do not wait on each other's hand-offs; each stream is ordered on
    // its own. All 32 lanes run the issue loop (waits are warp-uniform) and
    // one lane elected inside each instruction issues it: no branch around the
    // MMAs, whose operands then stay in uniform registers. Every ring entry
    // gets one release per slot: from the slot's softmax warps when the slot
    // runs in the unit, else from its issuer with a plain arrive once the
    // fill has landed.
    const int i = warp - kMmaWarp0;
    {
      constexpr uint32_t idesc_s = idesc_bf16_f32(128, kSub, false, false);  // Q, K both K-major
      constexpr uint32_t idesc_o = idesc_bf16_f32(128, D, false, true);      // V is MN-major (D contiguous)
      const uint32_t q_addr = smem_u32(sm.q[i]);
      const uint32_t s_tmem = tmem + 256 * i;
      // S_i(j) -> buffer b: Q_i [128 x D] times K sub-tile [64 x D]^T.
      auto issue_s = [&](int b, const uint8_t* ktile) {
        const uint32_t kaddr = smem_u32(ktile);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t qoff = (kk / 4) * kQBoxBytes + (kk % 4) * 32;
          const uint32_t koff = (kk / 4) * kKvBoxBytes + (kk % 4) * 32;
          mma_ss_elect(s_tmem + kSub * b, sdesc_sw128(q_addr + qoff, 16, 1024), sdesc_sw128(kaddr + koff, 16, 1024),
                 idesc_s, kk > 0);
        }
        mma_commit_elect(&sm.bar_s[i][b]);
      };
      // O_i (+)= P_i(j) [128 x 64, tensor memory] times V sub-tile [64 x D].
      // Only the unit's last two PVs signal their completion (bar_pvm, bar_o):
      // for the others, the completion of the score MMA issued after them does.
      auto issue_pv = [&](int b, const uint8_t* vtile, bool acc, uint64_t* done) {
        const uint32_t vaddr = smem_u32(vtile);
#pragma unroll
        for (int kk = 0; kk < kSub / 16; ++kk) {
          mma_ts_elect(s_tmem + 128, s_tmem + kSub * b + kk * 8, sdesc_sw128(vaddr + kk * 16 * 128, kKvBoxBytes, 1024),
                 idesc_o, (acc || kk > 0) ? 1u : 0u);
        }
        if (done) mma_commit_elect(done);
      };
      auto wait_fill = [&](int f) -> bool {
        return warp_wait(&sm.bar_full[f % kRing], (f / kRing) & 1, abort, p.err, p.wait_ns);
      };
      // A running slot's entries are released by its softmax warps, which see
      // the completion of the MMAs that read them (below); an idle slot
      // releases each entry once its fill has landed.
      auto release = [&](int f, bool issued) {
        if (!issued) mbar_arrive_elect(&sm.bar_empty[f % kRing]);
      };
      int q_loads = 0;    // bar_q phases consumed
      int units_run = 0;  // bar_ofree phases
      int p_seen = 0;     // bar_p hand-offs consumed
      int f = 0;          // ring fills consumed
      bool ok = true;
      for (int unit = blockIdx.x; ok && unit < p.units; unit += gridDim.x) {
        const Unit U = decode_unit<kMasked>(p, unit);
        if (U.nkv == 0) continue;
        const bool run = U.run[i];
        if (run) {
          ok = warp_wait(&sm.bar_q[i], q_loads & 1, abort, p.err, p.wait_ns);
          ++q_loads;
        }
        // Prologue: S(0) and S(1) into buffers 0 and 1 from the entry [K_0 | K_1].
        {
          const int fe = f++;
          if (!wait_fill(fe)) { ok = false; break; }
          if (run) {
            tc_fence_after();
            issue_s(0, sm.ring[fe % kRing][0]);
            if (U.nkv == 1) mma_commit_elect(&sm.bar_qfree[i]);
            if (U.nkv >= 2) {
              issue_s(1, sm.ring[fe % kRing][1]);
              if (U.nkv == 2) mma_commit_elect(&sm.bar_qfree[i]);
            }
          }
          release(fe, run);
        }
        // Step j: PV(j) from the entry's V_j, then S(j + 2) from its K_{j+2}.
        for (int j = 0; ok && j < U.nkv; ++j) {
          const int fe = f++;
          if (!wait_fill(fe)) { ok = false; break; }
          if (run) {
            // O_i of this slot's previous unit must have been read out before PV(0) overwrites it.
            if (j == 0 && units_run > 0 && !warp_wait(&sm.bar_ofree[i], (units_run - 1) & 1, abort, p.err, p.wait_ns)) {
              ok = false;
              break;
            }
            if (!warp_wait(&sm.bar_p[i][p_seen & 1], (p_seen >> 1) & 1, abort, p.err, p.wait_ns)) { ok = false; break; }
            ++p_seen;
            tc_fence_after();
            issue_pv(j & 1, sm.ring[fe % kRing][0], j > 0,
                     j == U.nkv - 1 ? &sm.bar_o[i] : (j == U.nkv - 2 ? &sm.bar_pvm[i] : nullptr));
            if (j + 2 < U.nkv) {
              issue_s(j & 1, sm.ring[fe % kRing][1]);
              if (j + 2 == U.nkv - 1) mma_commit_elect(&sm.bar_qfree[i]);
            }
          }
          release(fe, run);
        }
        if (run) ++units_run;
      }
      // Teardown: every MMA issued by this thread completes before TMEM is freed.
      mma_commit_elect(&sm.bar_done[i]);
      mbar_drain(&sm.bar_done[i], 0);
    }
    __syncwarp();
  } else {
    // ================================================================ softmax + epilogue
    const int i = warp >> 2;                 // tile slot
    const int qw = warp & 3;                 // warp within the warpgroup: rows 32 qw .. 32 qw + 31
    const int t = threadIdx.x & 127;         // row within the tile = TMEM lane
    const uint32_t lane_base = static_cast<uint32_t>(qw * 32) << 16;
    const uint32_t slot_addr = tmem + lane_base + 256 * i;
    const uint32_t o_addr = slot_addr + 128;
    uint32_t s_par = 0;      // bit b: parity of the next bar_s[i][b] phase
    // Ring entries of the running unit: [K_0 | K_1] at f0, [V_j | K_{j+2}] at
    // f0 + 1 + j. The MMAs of one issuer complete in order, so once S(x) has
    // completed so have PV(x - 2) and S(x), the readers of entry x - 2: one
    // thread per slot releases an entry when it sees that completion.
    int f_next = 0;          // ring entries of the units walked so far
    const bool rel_thread = t == 0;
    int unit_seq = 0;
    // PV completion: S(j) is issued after PV(j-2) and S(j+1) after PV(j-1)
    // (one issuer, in order), so waiting for a score buffer also waits for the
    // PVs before it. Only the unit's last two PVs have barriers of their own
    // (bar_pvm, bar_o), each consumed once per unit; their next phases need
    // hand-offs of the next unit, so they cannot run two phases ahead.
    uint32_t s_ahead = 0;    // bit b: the next phase of bar_s[i][b] already consumed
    int hand = 0;       // hand-offs so far: hand-off n on bar_p[i][n % 2]
    int pvm_seen = 0;   // bar_pvm phases consumed
    int units_run = 0;  // bar_o phases consumed
    bool ok = true;
    for (int unit = blockIdx.x; ok && unit < p.units; unit += gridDim.x) {
      const Unit U = decode_unit<kMasked>(p, unit);
      const int f0 = f_next;
      if (U.nkv > 0) f_next += U.nkv + 1;
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
      ++unit_seq;
      if (i == 1) {
        // Start slot 1 one softmax behind slot 0 so that the two slots' MMA
        // bursts alternate instead of coinciding.
        uint64_t t0 = global_timer_ns();
        while (*reinterpret_cast<volatile int*>(&sm.unit_flag) < unit_seq) {
          if (global_timer_ns() - t0 > p.wait_ns || *abort) { *abort = 1; ok = false; break; }
        }
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      }
      float m_used = -INFINITY;
      float l = 0.f;
      bool pvm_done = false;
      // This row's keys: [0, hi1) and [lo2, hi2).
      const KeyRanges kr = kMasked ? key_ranges(p.mask_mode, p.block, row, U.n, U.p) : KeyRanges{U.n, U.n, U.n};
      // S(x) seen complete: release the entry it and PV(x - 2) read.
      auto scores_seen = [&](int x) {
        if (!rel_thread) return;
        if (x >= 2) mbar_arrive(&sm.bar_empty[(f0 + x - 1) % kRing]);
        else if (x == 1 || U.nkv == 1) mbar_arrive(&sm.bar_empty[f0 % kRing]);
      };
      for (int j = 0; j < U.nkv; ++j) {
        const int b = j & 1;
        const uint32_t s_addr = slot_addr + kSub * b;
        if ((s_ahead >> b) & 1u) {
          s_ahead &= ~(1u << b);
        } else {
          if (!warp_wait(&sm.bar_s[i][b], (s_par >> b) & 1u, abort, p.err, p.wait_ns)) { ok = false; break; }
          s_par ^= 1u << b;
          scores_seen(j);
        }
        tc_fence_after();
        uint32_t sr[kSub];
        tmem_ld32(s_addr, *reinterpret_cast<uint32_t(*)[32]>(&sr[0]));
        tmem_ld32(s_addr + 32, *reinterpret_cast<uint32_t(*)[32]>(&sr[32]));
        tmem_wait_ld();
        float sv[kSub];
#pragma unroll
        for (int c = 0; c < kSub; ++c) sv[c] = __uint_as_float(sr[c]);
        const int key0 = (kMasked ? U.kt(j) : j) * kSub;
        if (!(key0 + kSub <= kr.hi1 || (kMasked && key0 >= kr.lo2 && key0 + kSub <= kr.hi2))) {
          // The row's keys in this sub-tile, [0, hi1) and [lo2, hi2), as bits;
          // one bit test per score.
          const uint64_t allow = key_bits(key0, 0, kr.hi1) | (kMasked ? key_bits(key0, kr.lo2, kr.hi2) : 0ull);
          const uint32_t alo = static_cast<uint32_t>(allow), ahi = static_cast<uint32_t>(allow >> 32);
#pragma unroll
          for (int c = 0; c < kSub; ++c) {
            if (!(((c < 32 ? alo : ahi) >> (c & 31)) & 1u)) sv[c] = -INFINITY;
          }
        }
        float mx0 = sv[0], mx1 = sv[1], mx2 = sv[2], mx3 = sv[3];
#pragma unroll
        for (int c = 4; c + 8 <= kSub; c += 8) {
          mx0 = fmax3(mx0, sv[c], sv[c + 1]);
          mx1 = fmax3(mx1, sv[c + 2], sv[c + 3]);
          mx2 = fmax3(mx2, sv[c + 4], sv[c + 5]);
          mx3 = fmax3(mx3, sv[c + 6], sv[c + 7]);
        }
        mx0 = fmax3(mx0, sv[kSub - 4], sv[kSub - 3]);
        mx1 = fmax3(mx1, sv[kSub - 2], sv[kSub - 1]);
        const float m_tile = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * p.scale_log2;
        const bool raise = m_tile > m_used + kRescaleThreshold;
        if (__any_sync(0xffffffffu, raise)) {
          const float m_new = raise ? m_tile : m_used;
          const float alpha = (m_used == -INFINITY) ? 0.f : ex2_approx(m_used - m_new);
          l *= alpha;
          m_used = m_new;
          if (j > 0) {
            // O holds sum_{j' < j} P V once PV(j-1) has completed: wait for the
            // score MMA issued after it (S(j+1)), or on the unit's last sub-tile
            // for PV(j-1)'s own barrier, then rescale.
            if (j + 1 < U.nkv) {
              const int bn = b ^ 1;
              if (!warp_wait(&sm.bar_s[i][bn], (s_par >> bn) & 1u, abort, p.err, p.wait_ns)) { ok = false; break; }
              s_par ^= 1u << bn;
              s_ahead |= 1u << bn;
              scores_seen(j + 1);
            } else {
              if (!warp_wait(&sm.bar_pvm[i], pvm_seen & 1, abort, p.err, p.wait_ns)) { ok = false; break; }
              ++pvm_seen;
              pvm_done = true;
              if (rel_thread) mbar_arrive(&sm.bar_empty[(f0 + U.nkv - 1) % kRing]);  // [V_{n-2}]
            }
            tc_fence_after();
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
        // Numerators 2^(s * scale - m), two columns at a time; P goes to tensor
        // memory (over the first 32 columns of this S buffer) 16 columns at a time.
        // The row sum l adds the numerators as rounded to bf16, the values the
        // PV product uses, so the output is an exactly normalised average of v
        // (a key that takes all the weight yields its v unchanged).
        const float2 sc2 = make_float2(p.scale_log2, p.scale_log2);
        // A row whose keys so far were all masked keeps m_used = -inf: its
        // numerators are exp2(-inf) = 0 (subtracting 0 avoids -inf - -inf).
        const float m_sub = (kMasked && m_used == -INFINITY) ? 0.f : m_used;
        const float2 nm2 = make_float2(-m_sub, -m_sub);
        float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
        for (int qq = 0; qq < kSub / 32; ++qq) {
          uint32_t pk[16];
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            const int col = 32 * qq + 2 * c;
            const float2 x = ffma2(make_float2(sv[col], sv[col + 1]), sc2, nm2);
            const float2 e = make_float2(ex2_approx(x.x), ex2_approx(x.y));
            pk[c] = pack_bf16x2(e.x, e.y);
            if (c & 1) acc1 = add_bf16x2_f32(acc1, pk[c]); else acc0 = add_bf16x2_f32(acc0, pk[c]);
          }
          tmem_st16(s_addr + 16 * qq, pk);
        }
        l += (acc0.x + acc0.y) + (acc1.x + acc1.y);
        tmem_wait_st();
        // Hand-off n uses bar_p[i][n % 2]; hand-off n + 2 comes after S(n + 2),
        // which the issuer starts only after consuming hand-off n.
        tc_fence_before();
        mbar_arrive(&sm.bar_p[i][hand & 1]);
        if (i == 0 && j == 0 && t == 0) *reinterpret_cast<volatile int*>(&sm.unit_flag) = unit_seq;
        ++hand;
      }
      // The unit's last two PVs (the next-to-last one only if not consumed above).
      if (ok && U.nkv >= 2 && !pvm_done) {
        if (!warp_wait(&sm.bar_pvm[i], pvm_seen & 1, abort, p.err, p.wait_ns)) ok = false;
        ++pvm_seen;
        if (ok && rel_thread) mbar_arrive(&sm.bar_empty[(f0 + U.nkv - 1) % kRing]);  // [V_{n-2}]
      }
      if (!ok || !warp_wait(&sm.bar_o[i], units_run & 1, abort, p.err, p.wait_ns)) { ok = false; break; }
      if (rel_thread) mbar_arrive(&sm.bar_empty[(f0 + U.nkv) % kRing]);  // [V_{n-1}]
      ++units_run;
      // Epilogue: read O_i out of tensor memory, hand the columns back to the
      // MMA warp, then normalise, convert to bf16, stage 32 rows x 32 columns
      // per warp in shared memory and write them with TMA stores (rows >= n
      // are zero; rows >= L are clipped by the tensor map). The staging rows
      // use the 64-byte swizzle of the output tensor map (16-byte chunk e of
      // row r at position e ^ ((r / 2) % 4)), which makes the warp's stores
      // free of shared-memory bank conflicts.
      tc_fence_after();
      const bool valid_row = row < U.n;
      const float inv = valid_row ? 1.0f / l : 0.f;
      const float2 inv2 = make_float2(inv, inv);
      // Rows >= n are written as zeros whatever O holds there (a NaN times
      // zero would not be zero).
      const uint32_t vmask = valid_row ? 0xFFFFFFFFu : 0u;
      const int wrow0 = U.row0[i] + 32 * qw;
      const bool store = wrow0 < p.L;
      if (store) {
        if (lane == 0) bulk_wait_read<0>();  // staging buffers of the previous unit are free
        __syncwarp();
      }
      // One 32-column chunk of O at a time (a compact loop: this code runs
      // once per unit); the columns go back to the MMA warp after the last.
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        uint32_t ov[32];
        tmem_ld32(o_addr + 32 * c, ov);
        tmem_wait_ld();
        if (c == D / 32 - 1) {
          tc_fence_before();
          mbar_arrive(&sm.bar_ofree[i]);
        }
        if (!store) continue;
        uint8_t* buf = sm.stage[warp][c & 1];
        if (c >= 2) {
          if (lane == 0) bulk_wait_read<1>();
          __syncwarp();
        }
        uint8_t* dstrow = buf + lane * 64;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          uint32_t w[4];
#pragma unroll
          for (int h = 0; h < 4; ++h) {
            const int col = 8 * e + 2 * h;
            const float2 x = fmul2(make_float2(__uint_as_float(ov[col]), __uint_as_float(ov[col + 1])), inv2);
            w[h] = pack_bf16x2(x.x, x.y) & vmask;
          }
          *reinterpret_cast<uint4*>(dstrow + ((e ^ ((lane >> 1) & 3)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_4d(&to, buf, 32 * c, U.head[i], wrow0, U.b);
          bulk_commit();
        }
      }
    }
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp0) {
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

template <int D, bool kMasked>
int launch_d(const AttnArgs& a, cudaStream_t stream) {
  CUtensorMap mq, mk, mv, mo;
  int st;
  if ((st = make_map(&mq, a.q, a.B, a.L, a.Hq, D, a.sq)) != DLM_OK) return st;
  if ((st = make_map(&mk, a.k, a.B, a.L, a.Hkv, D, a.sk, 64, kSub)) != DLM_OK) return st;
  if ((st = make_map(&mv, a.v, a.B, a.L, a.Hkv, D, a.sv, 64, kSub)) != DLM_OK) return st;
  // Output: 32 x 32 boxes (one warp's rows, one 64-byte column chunk), no swizzle.
  if ((st = make_map(&mo, a.out, a.B, a.L, a.Hq, D, a.so, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B)) != DLM_OK) return st;
  TcParams p;
  p.B = a.B;
  p.L = a.L;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.G = a.Hq / a.Hkv;
  p.mtiles = (a.L + kTile - 1) / kTile;
  // Two query tiles per work unit, one in each slot; one tile per unit only
  // when every tile then runs at once (twice the pairs still fit on the SMs:
  // a single short sequence). One-tile units take ~0.8 of a two-tile unit's
  // time, so a second round of them costs more than the pairs' one round
  // (measured at 1 x 512: 10.0 against 12.0 us; at 2 x 512: 17.2 against 12.8).
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long long pairs = static_cast<long long>(a.B) * a.Hkv * ((p.G * p.mtiles + 1) / 2);
  const int forced = attn_tiles_per_unit();
  p.tpu = forced ? forced : (2 * pairs <= sms ? 1 : 2);
  p.units_per_bg = (p.G * p.mtiles + p.tpu - 1) / p.tpu;
  p.div_upb = make_fastdiv(p.units_per_bg);
  p.div_hkv = make_fastdiv(p.Hkv);
  p.div_g = make_fastdiv(p.G);
  const long long units = static_cast<long long>(a.B) * a.Hkv * p.units_per_bg;
  if (units == 0) return DLM_OK;
  if (units > 0x7FFFFFFFLL) return fail(DLM_ERR_SHAPE, "too many attention work units");
  p.units = static_cast<int>(units);
  p.seq_lens = a.seq_lens;
  p.prompt_lens = a.prompt_lens;
  p.mask_mode = a.mask_mode;
  p.block = a.block > 0 ? a.block : 1;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.so0 = a.so[0];
  p.so1 = a.so[1];
  p.so2 = a.so[2];
  p.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(D));
  p.err = device_error_word();
  p.wait_ns = wait_budget_ns();
  const size_t smem = sizeof(Smem<D>) + 1024;
  cudaError_t attr_err = cudaFuncSetAttribute(attn_tc_kernel<D, kMasked>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              static_cast<int>(smem));
  if (attr_err != cudaSuccess) return fail(DLM_ERR_CUDA, "attn smem attribute: %s", cudaGetErrorString(attr_err));
  const int grid = static_cast<int>(units < sms ? units : sms);
  attn_tc_kernel<D, kMasked><<<grid, kThreads, smem, stream>>>(mq, mk, mv, mo, p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "attn_tc launch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

}  // namespace

int launch_attn_tc_bf16(const AttnArgs& a, cudaStream_t stream) {
  if (a.B == 0 || a.L == 0) return DLM_OK;
  if (a.mask_mode != DLM_ATTN_FULL)
    return a.D == 64 ? launch_d<64, true>(a, stream) : launch_d<128, true>(a, stream);
  return a.D == 64 ? launch_d<64, false>(a, stream) : launch_d<128, false>(a, stream);
}

}  // namespace dlm
