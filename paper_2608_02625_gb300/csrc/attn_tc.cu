// Step A1, bf16 path -- non-causal GQA attention on the 5th-generation tensor
// cores (tcgen05, accumulators in tensor memory, operands staged by TMA).
//
// Sec. 4.2: the refiner corrects over the entire sequence, so every valid
// query attends to every valid key (no causal or block mask); Sec. 3.3 is the
// block-causal pattern it replaces. out = softmax(q k^T / sqrt(D)) v per
// (sequence, query head), kv head = floor(h * Hkv / Hq), varlen via seq_lens.
//
// Work unit (one CTA): two 128-row query tiles that read the same key/value
// head of the same sequence (two query heads of one GQA group, or two row
// blocks of one head), so each 128-key K/V tile that TMA brings into shared
// memory feeds both. Warp roles (320 threads):
//   warps 0-3  softmax for tile slot 0 (thread t owns query row t = TMEM lane t)
//   warps 4-7  softmax for tile slot 1
//   warp 8     TMA producer (Q once, K/V through a 2-stage ring)
//   warp 9     tensor-memory allocator and MMA issuer (one elected thread)
// Tensor memory (512 columns x 128 lanes x 32 bit):
//   S_i = Q_i K_j^T  fp32, columns [128 i, 128 i + 128)
//   P_i = bf16 softmax numerators, written over the first 64 columns of S_i
//   O_i = sum_j P_i V_j fp32, columns [256 + D i, 256 + D i + D)
// MMA order per key tile j: PV_0(j), S_0(j+1), PV_1(j), S_1(j+1): the tensor
// core computes the next scores of one slot while the other slot's softmax
// runs. The tensor pipe executes one thread's tcgen05.mma in issue order, so
// S_i(j+1) overwrites P_i(j) only after PV_i(j) has read it.
// Online softmax in the log2 domain with exp2; the running maximum used for the
// numerators is raised (and O rescaled) only when it grows by more than 8,
// which bounds every numerator by 2^8 and leaves the final O / l exact.
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
constexpr int kStages = 2;          // K/V ring depth
constexpr int kThreads = 320;
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp = 9;
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D>
struct Smem {
  static constexpr int kBoxBytes = kTile * 64 * 2;     // one 128 x 64 bf16 TMA box (16 KB)
  static constexpr int kTileBytes = kTile * D * 2;     // D / 64 boxes
  alignas(1024) uint8_t q[2][kTileBytes];
  alignas(1024) uint8_t k[kStages][kTileBytes];
  alignas(1024) uint8_t v[kStages][kTileBytes];
  uint64_t bar_q;
  uint64_t bar_k[kStages];
  uint64_t bar_v[kStages];
  uint64_t bar_kv_empty[kStages];
  uint64_t bar_s[2];
  uint64_t bar_p[2];
  uint64_t bar_o[2];
  uint64_t bar_vtmp;
  uint64_t bar_done;
  uint32_t tmem_base;
  int abort;
};

struct TcParams {
  int B, L, Hq, Hkv, G, mtiles, units_per_bg;
  const int32_t* seq_lens;
  __nv_bfloat16* out;
  int64_t so0, so1, so2;
  float scale_log2;
  int* err;
};

// Warp-uniform bounded wait: true only if every lane saw the phase complete.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort, int* err) {
  bool ok = mbar_wait(bar, parity, abort, err);
  return __all_sync(0xffffffffu, ok);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tk,
                   const __grid_constant__ CUtensorMap tv, const TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  Smem<D>& sm = *reinterpret_cast<Smem<D>*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  constexpr int kBoxes = D / 64;
  constexpr uint32_t kBoxBytes = Smem<D>::kBoxBytes;
  constexpr uint32_t kTileBytes = Smem<D>::kTileBytes;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // ---- work unit
  const int unit = blockIdx.x;
  const int bg = unit / p.units_per_bg;
  const int u = unit % p.units_per_bg;
  const int b = bg / p.Hkv;
  const int g = bg % p.Hkv;
  int n = p.seq_lens ? p.seq_lens[b] : p.L;
  if (n < 0 || n > p.L) {
    if (threadIdx.x == 0) set_device_error(p.err, DLM_DEVERR_LENGTH);
    n = n < 0 ? 0 : p.L;
  }
  const int ntiles = p.G * p.mtiles;
  int head[2], row0[2];
  bool active[2], run[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int t = 2 * u + i;
    active[i] = t < ntiles;
    head[i] = g * p.G + (active[i] ? t % p.G : 0);
    row0[i] = (active[i] ? t / p.G : 0) * kTile;
    run[i] = active[i] && row0[i] < n;
  }
  const int nkv = (run[0] || run[1]) ? (n + kTile - 1) / kTile : 0;

  // ---- setup
  if (threadIdx.x == 0) {
    mbar_init(&sm.bar_q, 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.bar_k[s], 1);
      mbar_init(&sm.bar_v[s], 1);
      mbar_init(&sm.bar_kv_empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.bar_s[i], 1);
      mbar_init(&sm.bar_p[i], 128);
      mbar_init(&sm.bar_o[i], 1);
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
    int k_issued[kStages] = {0, 0}, v_issued[kStages] = {0, 0};
    bool q_issued = false, vtmp_issued = false;
    if (nkv > 0) {
      if (lane == 0) {
        prefetch_tmap(&tq);
        prefetch_tmap(&tk);
        prefetch_tmap(&tv);
        uint32_t qbytes = (run[0] ? kTileBytes : 0) + (run[1] ? kTileBytes : 0);
        mbar_arrive_expect_tx(&sm.bar_q, qbytes);
        for (int i = 0; i < 2; ++i)
          if (run[i])
            for (int c = 0; c < kBoxes; ++c)
              tma_load_4d(sm.q[i] + c * kBoxBytes, &tq, &sm.bar_q, 64 * c, head[i], row0[i], b);
      }
      q_issued = true;
      for (int j = 0; j < nkv; ++j) {
        const int s = j % kStages;
        if (j >= kStages && !warp_wait(&sm.bar_kv_empty[s], ((j / kStages) - 1) & 1, abort, p.err)) break;
        if (lane == 0) {
          mbar_arrive_expect_tx(&sm.bar_k[s], kTileBytes);
          for (int c = 0; c < kBoxes; ++c)
            tma_load_4d(sm.k[s] + c * kBoxBytes, &tk, &sm.bar_k[s], 64 * c, g, j * kTile, b);
        }
        ++k_issued[s];
        const int valid = n - j * kTile;
        if (valid >= kTile) {
          if (lane == 0) {
            mbar_arrive_expect_tx(&sm.bar_v[s], kTileBytes);
            for (int c = 0; c < kBoxes; ++c)
              tma_load_4d(sm.v[s] + c * kBoxBytes, &tv, &sm.bar_v[s], 64 * c, g, j * kTile, b);
          }
          ++v_issued[s];
        } else {
          // Last, partial tile: value rows >= n may hold any bit pattern and a
          // zero softmax weight does not cancel a NaN/Inf, so clear them in
          // shared memory before the MMA reads the tile.
          if (lane == 0) {
            mbar_arrive_expect_tx(&sm.bar_vtmp, kTileBytes);
            for (int c = 0; c < kBoxes; ++c)
              tma_load_4d(sm.v[s] + c * kBoxBytes, &tv, &sm.bar_vtmp, 64 * c, g, j * kTile, b);
          }
          vtmp_issued = true;
          if (!warp_wait(&sm.bar_vtmp, 0, abort, p.err)) break;
          const int zrows = kTile - valid;
          for (int c = 0; c < kBoxes; ++c) {
            uint4* base = reinterpret_cast<uint4*>(sm.v[s] + c * kBoxBytes + valid * 128);
            for (int e = lane; e < zrows * 8; e += 32) base[e] = make_uint4(0u, 0u, 0u, 0u);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.bar_v[s]);
          ++v_issued[s];  // completes one phase of bar_v[s], like a TMA fill
        }
      }
    }
    // Teardown: let every copy this warp issued land before the block exits.
    if (lane == 0) {
      if (q_issued) mbar_drain(&sm.bar_q, 0);
      if (vtmp_issued) mbar_drain(&sm.bar_vtmp, 0);
      for (int s = 0; s < kStages; ++s) {
        if (k_issued[s]) mbar_drain(&sm.bar_k[s], (k_issued[s] - 1) & 1);
        if (v_issued[s]) mbar_drain(&sm.bar_v[s], (v_issued[s] - 1) & 1);
      }
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ================================================================ MMA issuer
    if (lane == 0 && nkv > 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(128, 128, false, false);  // Q, K both K-major
      constexpr uint32_t idesc_o = idesc_bf16_f32(128, D, false, true);     // V is MN-major (D contiguous)
      const uint32_t q_addr[2] = {smem_u32(sm.q[0]), smem_u32(sm.q[1])};
      auto issue_s = [&](int i, int s) {
        const uint32_t kaddr = smem_u32(sm.k[s]);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk / 4) * kBoxBytes + (kk % 4) * 32;
          mma_ss(tmem + 128 * i, sdesc_sw128(q_addr[i] + off, 16, 1024),
                 sdesc_sw128(kaddr + off, 16, 1024), idesc_s, kk > 0);
        }
        mma_commit(&sm.bar_s[i]);
      };
      auto issue_pv = [&](int i, int s, bool acc) {
        const uint32_t vaddr = smem_u32(sm.v[s]);
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          mma_ts(tmem + 256 + D * i, tmem + 128 * i + kk * 8,
                 sdesc_sw128(vaddr + kk * 16 * 128, kBoxBytes, 1024), idesc_o, (acc || kk > 0) ? 1u : 0u);
        }
        mma_commit(&sm.bar_o[i]);
      };
      bool ok = mbar_wait(&sm.bar_q, 0, abort, p.err) && mbar_wait(&sm.bar_k[0], 0, abort, p.err);
      if (ok) {
        tc_fence_after();
        for (int i = 0; i < 2; ++i)
          if (run[i]) issue_s(i, 0);
      }
      for (int j = 0; ok && j < nkv; ++j) {
        const int s = j % kStages;
        const bool next = j + 1 < nkv;
        if (!mbar_wait(&sm.bar_v[s], (j / kStages) & 1, abort, p.err)) break;
        if (next && !mbar_wait(&sm.bar_k[(j + 1) % kStages], ((j + 1) / kStages) & 1, abort, p.err)) break;
        for (int i = 0; i < 2 && ok; ++i) {
          if (!run[i]) continue;
          if (!mbar_wait(&sm.bar_p[i], j & 1, abort, p.err)) { ok = false; break; }
          tc_fence_after();
          issue_pv(i, s, j > 0);
          if (next) issue_s(i, (j + 1) % kStages);
        }
        if (ok) mma_commit(&sm.bar_kv_empty[s]);
      }
    }
    if (lane == 0) {
      // Teardown: every MMA issued by this thread completes before TMEM is freed.
      mma_commit(&sm.bar_done);
      mbar_drain(&sm.bar_done, 0);
    }
    __syncwarp();
  } else {
    // ================================================================ softmax + epilogue
    const int i = warp >> 2;                 // tile slot
    const int t = threadIdx.x & 127;         // row within the tile = TMEM lane
    const uint32_t lane_base = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t s_addr = tmem + lane_base + 128 * i;
    const uint32_t o_addr = tmem + lane_base + 256 + D * i;
    const int row = row0[i] + t;
    bool ok = true;
    float l = 0.f;
    if (run[i]) {
      float m_used = -INFINITY;
      for (int j = 0; j < nkv; ++j) {
        if (!warp_wait(&sm.bar_s[i], j & 1, abort, p.err)) { ok = false; break; }
        tc_fence_after();
        uint32_t sr[128];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(s_addr + 32 * c, *reinterpret_cast<uint32_t(*)[32]>(&sr[32 * c]));
        tmem_wait_ld();
        float sv[128];
#pragma unroll
        for (int c = 0; c < 128; ++c) sv[c] = __uint_as_float(sr[c]);
        const int valid = n - j * kTile;
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
      if (ok) ok = warp_wait(&sm.bar_o[i], (nkv - 1) & 1, abort, p.err);
    }
    // Epilogue: out row = O / l (rows >= n are zero); skipped after a timeout.
    if (ok && active[i]) {
      const bool valid_row = run[i] && row < n;
      const float inv = valid_row ? 1.0f / l : 0.f;
      __nv_bfloat16* orow = p.out + b * p.so0 + static_cast<int64_t>(row) * p.so1 + head[i] * p.so2;
      if (run[i]) tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        uint32_t ov[32];
        if (run[i]) {
          tmem_ld32(o_addr + 32 * c, ov);
          tmem_wait_ld();
        }
        uint32_t pk[16];
#pragma unroll
        for (int e = 0; e < 16; ++e)
          pk[e] = valid_row ? pack_bf16x2(__uint_as_float(ov[2 * e]) * inv, __uint_as_float(ov[2 * e + 1]) * inv) : 0u;
        if (row < p.L) {
          uint4* dst = reinterpret_cast<uint4*>(orow + 32 * c);
#pragma unroll
          for (int e = 0; e < 4; ++e) dst[e] = make_uint4(pk[4 * e], pk[4 * e + 1], pk[4 * e + 2], pk[4 * e + 3]);
        }
      }
    }
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
// box = 64 head-dim elements x 1 head x 128 rows x 1 sequence, 128-byte swizzle.
int make_map(CUtensorMap* map, const void* base, int B, int L, int H, int D, const int64_t* s) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return fail(DLM_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(H), static_cast<cuuint64_t>(L),
                        static_cast<cuuint64_t>(B)};
  cuuint64_t strides[3] = {static_cast<cuuint64_t>(s[2]) * 2, static_cast<cuuint64_t>(s[1]) * 2,
                           static_cast<cuuint64_t>(s[0]) * 2};
  cuuint32_t box[4] = {64, 1, kTile, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(DLM_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return DLM_OK;
}

template <int D>
int launch_d(const AttnArgs& a, cudaStream_t stream) {
  CUtensorMap mq, mk, mv;
  int st;
  if ((st = make_map(&mq, a.q, a.B, a.L, a.Hq, D, a.sq)) != DLM_OK) return st;
  if ((st = make_map(&mk, a.k, a.B, a.L, a.Hkv, D, a.sk)) != DLM_OK) return st;
  if ((st = make_map(&mv, a.v, a.B, a.L, a.Hkv, D, a.sv)) != DLM_OK) return st;
  TcParams p;
  p.B = a.B;
  p.L = a.L;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.G = a.Hq / a.Hkv;
  p.mtiles = (a.L + kTile - 1) / kTile;
  p.units_per_bg = (p.G * p.mtiles + 1) / 2;
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
  const long long units = static_cast<long long>(a.B) * a.Hkv * p.units_per_bg;
  if (units == 0) return DLM_OK;
  attn_tc_kernel<D><<<static_cast<unsigned>(units), kThreads, smem, stream>>>(mq, mk, mv, p);
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
