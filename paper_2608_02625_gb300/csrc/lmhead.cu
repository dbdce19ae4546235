// The vocabulary projection fused with step A2, on the tensor cores.
//
// Every revisable position's distribution over the vocabulary comes from the
// refiner's output projection of its final hidden state (Sec. 4.2):
// logits[r, v] = hidden[r, :] . weight[v, :]. This kernel computes, per row,
// what the vocabulary reduction of those logits computes (argmax with ties to
// the lowest index, maximum softmax probability, log-sum-exp) without ever
// writing the N x V logits to memory.
//
// Persistent CTAs (one per SM) walk work items = (vocabulary split, block of
// 128 rows); items are ordered split-major, so the CTAs running at the same
// time read the same weight tiles and those stay in L2. Per 128 x 256 output
// tile:
//   warp 0     TMA producer: hidden box 128 x 64 and weight box 256 x 64 per
//              64-wide K step, through a 4-stage ring (48 KB a stage)
//   warp 1     tensor-memory allocator and MMA issuer (all lanes run the loop,
//              one lane elected per instruction):
//              tcgen05.mma kind::f16, M = 128, N = 256, K = 16, bf16 x bf16 ->
//              fp32 accumulators; two accumulators of 256 columns, so the
//              epilogue of a tile overlaps the K loop of the next
//   warps 4-7  epilogue: thread t owns row t (TMEM lane t); 32 columns at a
//              time it takes the chunk's maximum and first index, rescales its
//              running sum of exp(x - m) when the maximum grows, and adds the
//              chunk's terms (per-tile partial sums keep the fp32 sum short)
// At the end of an item each row's (max, first index, sum) is written to the
// caller's workspace; lmhead_combine_kernel merges the splits of a row in
// vocabulary order (ties keep the lower index). Every mbarrier wait is
// bounded; on expiry the kernel sets DLM_DEVERR_TIMEOUT, drains and exits.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "dlm_common.cuh"
#include "dlm_internal.h"

namespace dlm {
namespace {

constexpr int kBM = 128;          // rows per tile = TMEM lanes
constexpr int kBN = 256;          // vocabulary columns per tile
constexpr int kBK = 64;           // K per stage: one 128-byte swizzle atom of bf16
constexpr int kStages = 4;
constexpr int kThreads = 256;     // warp 0 TMA, warp 1 MMA, warps 4-7 epilogue
constexpr int kEpiWarp0 = 4;
constexpr uint32_t kTmemCols = 512;
constexpr int kABytes = kBM * kBK * 2;  // 16 KB
constexpr int kBBytes = kBN * kBK * 2;  // 32 KB
constexpr float kLog2e = 1.4426950408889634f;

struct Smem {
  alignas(1024) uint8_t a[kStages][kABytes];
  alignas(1024) uint8_t b[kStages][kBBytes];
  uint64_t full[kStages];     // stage loaded             (TMA -> MMA)
  uint64_t empty[kStages];    // stage read by its MMAs   (MMA -> TMA)
  uint64_t acc_full[2];       // accumulator complete     (MMA -> epilogue)
  uint64_t acc_empty[2];      // accumulator read out     (epilogue -> MMA)
  uint64_t done;              // every MMA completed      (teardown)
  uint32_t tmem_base;
  int abort;
};

struct LmParams {
  int N, V, d;
  int row_blocks, vtiles, splits, items;
  float* part_m;
  int* part_idx;
  float* part_s;
  int* err;
  uint64_t wait_ns;  // budget of each bounded wait
};

struct Item {
  int rb, split, t0, t1;  // row block, split, vocabulary tiles [t0, t1)
};

__device__ __forceinline__ Item item_at(const LmParams& p, int item) {
  Item it;
  it.split = item / p.row_blocks;
  it.rb = item % p.row_blocks;
  it.t0 = static_cast<int>(static_cast<long long>(p.vtiles) * it.split / p.splits);
  it.t1 = static_cast<int>(static_cast<long long>(p.vtiles) * (it.split + 1) / p.splits);
  return it;
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort, int* err,
                                          uint64_t budget_ns) {
  bool ok = mbar_wait_for(bar, parity, abort, err, budget_ns);
  return __all_sync(0xffffffffu, ok);
}

__global__ void __launch_bounds__(kThreads, 1)
    lmhead_kernel(const __grid_constant__ CUtensorMap th, const __grid_constant__ CUtensorMap tw, const LmParams p) {
  extern __shared__ uint8_t smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int kblocks = p.d / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.acc_full[i], 1);
      mbar_init(&sm.acc_empty[i], 128);
    }
    mbar_init(&sm.done, 1);
    sm.abort = 0;
    fence_mbar_init();
    fence_proxy_async_smem();
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  volatile int* abort = &sm.abort;

  if (warp == 0) {
    // ================================================================ TMA producer
    if (lane == 0) {
      prefetch_tmap(&th);
      prefetch_tmap(&tw);
    }
    int fill = 0;
    bool ok = true;
    for (int item = blockIdx.x; ok && item < p.items; item += gridDim.x) {
      const Item it = item_at(p, item);
      for (int vt = it.t0; ok && vt < it.t1; ++vt) {
        for (int kb = 0; kb < kblocks; ++kb, ++fill) {
          const int st = fill % kStages;
          if (fill >= kStages && !warp_wait(&sm.empty[st], ((fill / kStages) - 1) & 1, abort, p.err, p.wait_ns)) {
            ok = false;
            break;
          }
          if (lane == 0) {
            mbar_arrive_expect_tx(&sm.full[st], kABytes + kBBytes);
            tma_load_2d(sm.a[st], &th, &sm.full[st], kb * kBK, it.rb * kBM);
            tma_load_2d(sm.b[st], &tw, &sm.full[st], kb * kBK, vt * kBN);
          }
        }
      }
    }
    // Teardown: every copy issued lands before the block exits.
    if (lane == 0) {
      for (int s = 0; s < kStages; ++s) {
        const int n_s = fill > s ? (fill - s + kStages - 1) / kStages : 0;
        if (n_s) mbar_drain(&sm.full[s], (n_s - 1) & 1);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ================================================================ MMA issuer
    // All 32 lanes run the loop (warp-uniform waits); one lane elected inside
    // each MMA / commit issues it, with no branch around the MMAs.
    {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, kBN, false, false);  // both operands K-major
      int fill = 0, tile = 0;
      bool ok = true;
      for (int item = blockIdx.x; ok && item < p.items; item += gridDim.x) {
        const Item it = item_at(p, item);
        for (int vt = it.t0; ok && vt < it.t1; ++vt, ++tile) {
          const int acc = tile & 1;
          // The accumulator's previous tile (tile - 2) must have been read out.
          if (tile >= 2 && !warp_wait(&sm.acc_empty[acc], ((tile >> 1) - 1) & 1, abort, p.err, p.wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem + acc * kBN;
          for (int kb = 0; kb < kblocks; ++kb, ++fill) {
            const int st = fill % kStages;
            if (!warp_wait(&sm.full[st], (fill / kStages) & 1, abort, p.err, p.wait_ns)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a_addr = smem_u32(sm.a[st]);
            const uint32_t b_addr = smem_u32(sm.b[st]);
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk)
              mma_ss_elect(d_tmem, sdesc_sw128(a_addr + kk * 32, 16, 1024), sdesc_sw128(b_addr + kk * 32, 16, 1024),
                           idesc, (kb > 0 || kk > 0) ? 1u : 0u);
            mma_commit_elect(&sm.empty[st]);
          }
          if (!ok) break;
          mma_commit_elect(&sm.acc_full[acc]);
        }
      }
      mma_commit_elect(&sm.done);
      mbar_drain(&sm.done, 0);
    }
    __syncwarp();
  } else if (warp >= kEpiWarp0) {
    // ================================================================ epilogue
    const int qw = warp - kEpiWarp0;                 // TMEM lanes 32 qw .. 32 qw + 31
    const int t = threadIdx.x - kEpiWarp0 * 32;      // row within the tile
    const uint32_t lane_base = static_cast<uint32_t>(qw * 32) << 16;
    int tile = 0;
    bool ok = true;
    for (int item = blockIdx.x; ok && item < p.items; item += gridDim.x) {
      const Item it = item_at(p, item);
      float m = -INFINITY, s = 0.f;
      int idx = 0;
      for (int vt = it.t0; vt < it.t1; ++vt, ++tile) {
        const int acc = tile & 1;
        if (!warp_wait(&sm.acc_full[acc], (tile >> 1) & 1, abort, p.err, p.wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t base = tmem + lane_base + acc * kBN;
        float ts = 0.f;  // this tile's terms, relative to m
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) {
          uint32_t v[32];
          tmem_ld32(base + 32 * c, v);
          tmem_wait_ld();
          if (c == kBN / 32 - 1) {
            tc_fence_before();
            mbar_arrive(&sm.acc_empty[acc]);  // every column of the accumulator has been read
          }
          const int col0 = vt * kBN + 32 * c;
          float x[32];
          float cm = -INFINITY;
          int ci = 0;
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            x[e] = col0 + e < p.V ? __uint_as_float(v[e]) : -INFINITY;
            if (x[e] > cm) {
              cm = x[e];
              ci = col0 + e;
            }
          }
          if (cm > m) {
            const float a = m == -INFINITY ? 0.f : ex2_approx((m - cm) * kLog2e);
            s *= a;
            ts *= a;
            m = cm;
            idx = ci;
          }
          if (m != -INFINITY) {
            const float ml = m * kLog2e;
            float c0 = 0.f, c1 = 0.f;
#pragma unroll
            for (int e = 0; e < 32; e += 2) {
              c0 += ex2_approx(fmaf(x[e], kLog2e, -ml));
              c1 += ex2_approx(fmaf(x[e + 1], kLog2e, -ml));
            }
            ts += c0 + c1;
          }
        }
        s += ts;
      }
      if (!ok) break;
      const int row = it.rb * kBM + t;
      if (row < p.N) {
        const int64_t o = static_cast<int64_t>(it.split) * p.N + row;
        p.part_m[o] = m;
        p.part_idx[o] = idx;
        p.part_s[o] = s;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Merges the splits of each row in vocabulary order.
__global__ void lmhead_combine_kernel(const float* part_m, const int* part_idx, const float* part_s, int N,
                                      int splits, int32_t* argmax, float* conf, float* lse) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= N) return;
  float m = -INFINITY, s = 0.f;
  int idx = 0;
  for (int k = 0; k < splits; ++k) {
    const int64_t o = static_cast<int64_t>(k) * N + r;
    const float mk = part_m[o];
    const float sk = part_s[o];
    if (mk > m) {
      s = (m == -INFINITY ? 0.f : s * expf(m - mk)) + sk;
      m = mk;
      idx = part_idx[o];
    } else if (mk != -INFINITY) {
      s += sk * expf(mk - m);
    }
  }
  argmax[r] = idx;
  conf[r] = 1.0f / s;
  lse[r] = m + logf(s);
}

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

// 2-D map over a [rows, d] bf16 matrix (row stride in elements), box d 64 x box_rows.
int make_map_2d(CUtensorMap* map, const void* base, int64_t rows, int d, int64_t row_stride, int box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return fail(DLM_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(row_stride) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(DLM_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return DLM_OK;
}

}  // namespace

int lmhead_splits(int64_t N, int64_t V, int sms) {
  const int64_t row_blocks = (N + kBM - 1) / kBM;
  const int64_t vtiles = (V + kBN - 1) / kBN;
  int best = 1;
  double best_cost = 1e300;
  for (int s = 1; s <= kLmMaxSplits && s <= vtiles; ++s) {
    const int64_t items = row_blocks * s;
    const int64_t rounds = (items + sms - 1) / sms;
    // Tiles on the busiest CTA, plus a small cost per item (pipeline fill, flush).
    const double cost = static_cast<double>(rounds) * (static_cast<double>((vtiles + s - 1) / s) + 0.5);
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best = s;
    }
  }
  return best;
}

int launch_lmhead(const LmArgs& a, cudaStream_t stream) {
  if (a.N == 0) return DLM_OK;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  LmParams p;
  p.N = static_cast<int>(a.N);
  p.V = static_cast<int>(a.V);
  p.d = static_cast<int>(a.d);
  p.row_blocks = static_cast<int>((a.N + kBM - 1) / kBM);
  p.vtiles = static_cast<int>((a.V + kBN - 1) / kBN);
  p.splits = lmhead_splits(a.N, a.V, sms);
  p.items = p.row_blocks * p.splits;
  float* ws = static_cast<float*>(a.workspace);
  p.part_m = ws;
  p.part_idx = reinterpret_cast<int*>(ws + static_cast<int64_t>(p.splits) * a.N);
  p.part_s = ws + 2 * static_cast<int64_t>(p.splits) * a.N;
  p.err = device_error_word();
  p.wait_ns = wait_budget_ns();
  CUtensorMap mh, mw;
  int st;
  if ((st = make_map_2d(&mh, a.hidden, a.N, p.d, a.s_hidden, kBM)) != DLM_OK) return st;
  if ((st = make_map_2d(&mw, a.weight, a.V, p.d, a.s_weight, kBN)) != DLM_OK) return st;
  const size_t smem = sizeof(Smem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(lmhead_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "lmhead smem attribute: %s", cudaGetErrorString(e));
  const int grid = p.items < sms ? p.items : sms;
  lmhead_kernel<<<grid, kThreads, smem, stream>>>(mh, mw, p);
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "lmhead launch: %s", cudaGetErrorString(e));
  lmhead_combine_kernel<<<static_cast<unsigned>((a.N + 255) / 256), 256, 0, stream>>>(
      p.part_m, p.part_idx, p.part_s, p.N, p.splits, a.argmax, a.conf, a.lse);
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(DLM_ERR_CUDA, "lmhead combine launch: %s", cudaGetErrorString(e));
  return DLM_OK;
}

}  // namespace dlm
