// qkv_rope.cu -- fused QKV projection + rotary embedding + KV-cache append.
//
// Sec. 3.2 / Eq. 1: besides attention, each chunk pays GEMM work that grows
// with its length alone (QKV projection, output projection, FFN).  This is
// the first of those GEMMs, fused with what the attention needs next:
//   [Q | K | V] = X W^T                     (X [len, hidden], W [Nout, hidden])
//   Q, K rotated by RoPE at positions offset + r (rotate-half convention:
//     dims j and j + d/2 of a head turn by pos * theta^(-2j/d))
//   The angle is formed in integer fixed point, in turns: the host gives
//   step_j = theta^(-2j/d) / (2 pi) as a 64-bit binary fraction, and
//   pos * step_j modulo 2^64 is the angle's fraction of a full turn exactly
//   up to step_j's rounding (2^-64), with no floating-point reduction; its
//   top 32 bits, read as a signed integer, give the angle in [-pi, pi).
//   Q -> q_out [len, Hq, d];  K, V -> cache rows [offset, offset + len)
//
// Persistent warp-specialised tcgen05 GEMM, one CTA per SM:
//   warp 0      TMA producer: A = X tile [128 x 64], B = W tile [256 x 64]
//               per K step through a 4-stage ring (48 KB per stage)
//   warp 1      MMA issuer (converged warp, elected lane): M=128, N=256,
//               K=16 steps into one of two TMEM accumulators (2 x 256 cols)
//   warps 2-5   epilogue: thread r owns TMEM lane r = output row r; fp32 ->
//               RoPE (Q, K) -> bf16 -> 16-byte stores; the second accumulator
//               lets the next tile's main loop run during this epilogue.
// Tiles are visited with the row tile fastest so CTAs resident together
// share the same weight tile in L2.
#include <cmath>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "internal.h"
#include "sm103_ptx.cuh"

namespace mocap {
namespace {

constexpr int kBM = 128, kBN = 256, kBK = 64;
#ifndef MOCAP_QKV_STAGES
#define MOCAP_QKV_STAGES 4
#endif
constexpr int kStages = MOCAP_QKV_STAGES;
constexpr int kThreads = 192;  // 6 warps
constexpr int kABytes = kBM * kBK * 2;  // 16 KB
constexpr int kBBytes = kBN * kBK * 2;  // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kMaxHalfDim = 64;         // d <= 128

struct QkvParams {
  CUtensorMap tx;  // X [len, hidden], box {64, 128}
  CUtensorMap tw;  // W [Nout, hidden], box {64, 256}
  __nv_bfloat16 *q_out;
  __nv_bfloat16 *k_cache;  // already offset to row `offset`
  __nv_bfloat16 *v_cache;
  uint32_t *status;
  int64_t pos0;            // position of row 0
  int32_t len, hidden, n_q_heads, n_kv_heads, head_dim;
  int32_t m_tiles, n_tiles, k_steps;
  uint64_t turn_step[kMaxHalfDim];  // theta^(-2j/d) / (2 pi) * 2^64, rounded down
};

struct QkvLayout {
  static constexpr int kRing = 0;
  static constexpr int kBars = kStages * kStageBytes;
  // full[S], empty[S], acc_full[2], acc_empty[2], drain
  static constexpr int kBarFull = 0, kBarEmpty = kStages, kBarAccFull = 2 * kStages,
                       kBarAccEmpty = 2 * kStages + 2, kBarDrain = 2 * kStages + 4,
                       kNumBars = 2 * kStages + 5;
  static constexpr int kTmemSlot = kBars + 8 * kNumBars;
  static constexpr int kBytes = kTmemSlot + 8 + 1024;
};
static_assert(QkvLayout::kBytes <= 232448, "shared memory");

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// Epilogue for one head's d columns of one row: RoPE (if `rotate`), bf16,
// stores.  `taddr` is this lane's TMEM address of the head's first column.
template <int D>
__device__ __forceinline__ void emit_head(uint32_t taddr, bool rotate, uint64_t pos,
                                          const uint64_t *turn_step, __nv_bfloat16 *dst,
                                          bool valid) {
  constexpr int H = D / 2;
#pragma unroll
  for (int c = 0; c < H; c += 32) {
    uint32_t lo[32], hi[32];
    tmem_ld32(taddr + c, lo);       // dims c .. c+31
    tmem_ld32(taddr + H + c, hi);   // dims H+c .. H+c+31
    float a[32], b[32];
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      a[e] = __uint_as_float(lo[e]);
      b[e] = __uint_as_float(hi[e]);
    }
    if (rotate) {
#pragma unroll 4
      for (int e = 0; e < 32; ++e) {
        // fraction of a turn, modulo 1 by the wrap-around of the product
        const uint64_t turns = pos * turn_step[c + e];
        const float ang = static_cast<float>(static_cast<int32_t>(turns >> 32)) *
                          1.46291807926715968e-9f;  // 2 pi / 2^32
        float sn, cs;
        __sincosf(ang, &sn, &cs);
        const float x0 = a[e], x1 = b[e];
        a[e] = x0 * cs - x1 * sn;
        b[e] = x1 * cs + x0 * sn;
      }
    }
    if (valid) {
      uint4 *d0 = reinterpret_cast<uint4 *>(dst + c);
      uint4 *d1 = reinterpret_cast<uint4 *>(dst + H + c);
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        d0[v] = make_uint4(pack2(a[8 * v], a[8 * v + 1]), pack2(a[8 * v + 2], a[8 * v + 3]),
                           pack2(a[8 * v + 4], a[8 * v + 5]), pack2(a[8 * v + 6], a[8 * v + 7]));
        d1[v] = make_uint4(pack2(b[8 * v], b[8 * v + 1]), pack2(b[8 * v + 2], b[8 * v + 3]),
                           pack2(b[8 * v + 4], b[8 * v + 5]), pack2(b[8 * v + 6], b[8 * v + 7]));
      }
    }
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1) qkv_rope_kernel(const __grid_constant__ QkvParams p) {
  using L = QkvLayout;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t *gbase = smem_raw + (base - raw);
  const uint32_t bars = base + L::kBars;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };
  volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(gbase + L::kTmemSlot);
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31u;

  __shared__ uint32_t abort_flag;
  if (threadIdx.x == 0) abort_flag = *reinterpret_cast<volatile uint32_t *>(p.status);
  __syncthreads();
  if (abort_flag != 0u) return;

  if (warp == 1) {
    tmem_alloc(base + L::kTmemSlot, 512);
    tmem_relinquish();
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(bar(L::kBarFull + s), 1);
      mbar_init(bar(L::kBarEmpty + s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar(L::kBarAccFull + b), 1);
      mbar_init(bar(L::kBarAccEmpty + b), 4);  // one arrive per epilogue warp
    }
    mbar_init(bar(L::kBarDrain), 1);
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int n_tiles_total = p.m_tiles * p.n_tiles;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&p.tx);
      prefetch_tmap(&p.tw);
      int it = 0;  // global K-step counter across tiles (ring position)
      bool ok = true;
      for (int t = blockIdx.x; t < n_tiles_total && ok; t += gridDim.x) {
        const int mt = t % p.m_tiles, nt = t / p.m_tiles;
        for (int ks = 0; ks < p.k_steps; ++ks, ++it) {
          const int st = it % kStages;
          if (it >= kStages &&
              !mbar_wait(bar(L::kBarEmpty + st), ((it / kStages) - 1) & 1, p.status, kWaitLimitNs,
                         true, kHintProducer)) {
            ok = false;
            break;
          }
          const uint32_t sa = base + L::kRing + st * kStageBytes;
          mbar_arrive_expect_tx(bar(L::kBarFull + st), kStageBytes);
          tma_load_2d(sa, &p.tx, bar(L::kBarFull + st), ks * kBK, mt * kBM);
          tma_load_2d(sa + kABytes, &p.tw, bar(L::kBarFull + st), ks * kBK, nt * kBN);
        }
      }
      // copies in flight land before exit; last releases observed
      const int first = max(0, it - kStages);
      for (int s2 = first; s2 < it; ++s2)
        mbar_wait(bar(L::kBarFull + s2 % kStages), (s2 / kStages) & 1, p.status, 20000000ull,
                  false);
      if (ok)
        for (int s2 = first; s2 < it; ++s2)
          if (!mbar_wait(bar(L::kBarEmpty + s2 % kStages), (s2 / kStages) & 1, p.status)) break;
    }
  } else if (warp == 1) {
    const bool leader = elect_one();
    constexpr uint32_t idesc = idesc_bf16_f32(kBM, kBN, false, false);
    const uint64_t a0 = sdesc_sw128(base + L::kRing, 16, 1024);
    const uint64_t b0 = sdesc_sw128(base + L::kRing + kABytes, 16, 1024);
    constexpr uint64_t kStageStep = static_cast<uint64_t>(kStageBytes >> 4);
    int it = 0, tile_i = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles_total && ok; t += gridDim.x, ++tile_i) {
      const int buf = tile_i & 1;
      const int use = tile_i >> 1;  // how often this buffer was used before
      if (use > 0) ok = mbar_wait_warp(bar(L::kBarAccEmpty + buf), (use - 1) & 1, p.status, 0);
      if (!ok) break;
      tc_fence_after();
      const uint32_t acc = tmem + buf * kBN;
      for (int ks = 0; ks < p.k_steps; ++ks, ++it) {
        const int st = it % kStages;
        ok = mbar_wait_warp(bar(L::kBarFull + st), (it / kStages) & 1, p.status, 0);
        if (!ok) break;
        tc_fence_after();
        if (leader) {
          const uint64_t ad = a0 + st * kStageStep, bd = b0 + st * kStageStep;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)
            mma_ss(acc, ad + 2 * kk, bd + 2 * kk, idesc, (ks > 0 || kk > 0) ? 1u : 0u);
          tc_commit(bar(L::kBarEmpty + st));
        }
        __syncwarp();
      }
      if (!ok) break;
      if (leader) tc_commit(bar(L::kBarAccFull + buf));
      __syncwarp();
    }
    if (leader) {  // every issued MMA completes before TMEM is released
      tc_commit(bar(L::kBarDrain));
      mbar_wait(bar(L::kBarDrain), 0, p.status, 20000000ull, false);
    }
    __syncwarp();
  } else {
    // epilogue warps 2..5: TMEM lane quarter = warp % 4
    const uint32_t quarter = warp & 3u;
    const int row_in_tile = static_cast<int>(quarter * 32 + lane);
    const uint32_t lane_addr = tmem + ((quarter * 32u) << 16);
    const int q_cols = p.n_q_heads * D, k_cols = p.n_kv_heads * D;
    int tile_i = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles_total && ok; t += gridDim.x, ++tile_i) {
      const int buf = tile_i & 1;
      const int use = tile_i >> 1;
      ok = mbar_wait_warp(bar(L::kBarAccFull + buf), use & 1, p.status, kHintSoftmax);
      if (!ok) break;
      tc_fence_after();
      const int mt = t % p.m_tiles, nt = t / p.m_tiles;
      const int row = mt * kBM + row_in_tile;
      const bool valid = row < p.len;
      const uint64_t pos = static_cast<uint64_t>(p.pos0 + row);
#pragma unroll 1
      for (int hs = 0; hs < kBN / D; ++hs) {
        const int col = nt * kBN + hs * D;  // first output feature of this head
        __nv_bfloat16 *dst;
        bool rotate = true;
        if (col < q_cols) {
          dst = p.q_out + (static_cast<int64_t>(row) * p.n_q_heads + col / D) * D;
        } else if (col < q_cols + k_cols) {
          dst = p.k_cache + (static_cast<int64_t>(row) * p.n_kv_heads + (col - q_cols) / D) * D;
        } else {
          dst = p.v_cache +
                (static_cast<int64_t>(row) * p.n_kv_heads + (col - q_cols - k_cols) / D) * D;
          rotate = false;
        }
        emit_head<D>(lane_addr + buf * kBN + hs * D, rotate, pos, p.turn_step, dst, valid);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(L::kBarAccEmpty + buf));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn2() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 2-D bf16 [rows, cols] row-major, box {64 cols, box_rows}, 128-byte swizzle.
bool make_map_2d(CUtensorMap *map, const void *ptr, int64_t rows, int64_t cols, int box_rows) {
  auto fn = encode_fn2();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t elem[2] = {1u, 1u};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box,
            elem, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count_qkv() {
  static int cached[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (cached[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 148;
    cached[dev] = n;
  }
  return cached[dev];
}

}  // namespace
}  // namespace mocap

extern "C" mocap_status mocap_qkv_rope_append(const void *x, const void *w_qkv, void *q_out,
                                              void *k_cache, void *v_cache,
                                              int64_t cache_capacity, int64_t offset, int64_t len,
                                              int32_t hidden, int32_t n_q_heads,
                                              int32_t n_kv_heads, int32_t head_dim,
                                              float rope_theta, mocap_stream_t stream) {
  using namespace mocap;
  if (!x || !w_qkv || !q_out || !k_cache || !v_cache) return MOCAP_EINVAL;
  if (!aligned16(x) || !aligned16(w_qkv) || !aligned16(q_out) || !aligned16(k_cache) ||
      !aligned16(v_cache))
    return MOCAP_EINVAL;
  if (n_q_heads < 1 || n_kv_heads < 1 || n_q_heads % n_kv_heads != 0) return MOCAP_EINVAL;
  if (head_dim != 64 && head_dim != 128) return MOCAP_EUNSUPPORTED;
  if (hidden < 8 || hidden % 8 != 0) return MOCAP_EINVAL;  // 16-byte row stride for TMA
  if (offset < 0 || len < 0 || cache_capacity < 0 || offset > cache_capacity ||
      len > cache_capacity - offset || offset + len > 0x7fffffffLL)
    return MOCAP_EINVAL;
  if (!(rope_theta > 1.0f) || !std::isfinite(rope_theta)) return MOCAP_EINVAL;
  const int64_t n_out = static_cast<int64_t>(n_q_heads + 2 * n_kv_heads) * head_dim;
  if (n_out % kBN != 0) return MOCAP_EUNSUPPORTED;  // whole 256-column tiles
  if (len == 0) return MOCAP_OK;
  uint32_t *status = device_status_ptr();
  if (status == nullptr) return MOCAP_ECUDA;

  static QkvParams prm;
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  std::memset(&prm, 0, sizeof(prm));
  if (!make_map_2d(&prm.tx, x, len, hidden, kBM) || !make_map_2d(&prm.tw, w_qkv, n_out, hidden, kBN))
    return MOCAP_ECUDA;
  const size_t kv_row = static_cast<size_t>(n_kv_heads) * head_dim;
  prm.q_out = static_cast<__nv_bfloat16 *>(q_out);
  prm.k_cache = static_cast<__nv_bfloat16 *>(k_cache) + static_cast<size_t>(offset) * kv_row;
  prm.v_cache = static_cast<__nv_bfloat16 *>(v_cache) + static_cast<size_t>(offset) * kv_row;
  prm.status = status;
  prm.pos0 = offset;
  prm.len = static_cast<int32_t>(len);
  prm.hidden = hidden;
  prm.n_q_heads = n_q_heads;
  prm.n_kv_heads = n_kv_heads;
  prm.head_dim = head_dim;
  prm.m_tiles = static_cast<int32_t>((len + kBM - 1) / kBM);
  prm.n_tiles = static_cast<int32_t>(n_out / kBN);
  prm.k_steps = (hidden + kBK - 1) / kBK;
  for (int j = 0; j < head_dim / 2; ++j) {
    const double turns = std::pow(static_cast<double>(rope_theta), -2.0 * j / head_dim) /
                         6.283185307179586477;  // < 1/(2 pi): fits below 2^62 once scaled
    prm.turn_step[j] = static_cast<uint64_t>(std::ldexp(turns, 64));
  }

  const int64_t tiles = static_cast<int64_t>(prm.m_tiles) * prm.n_tiles;
  const int grid = static_cast<int>(std::min<int64_t>(tiles, sm_count_qkv()));
  auto launch = [&](auto kern) -> mocap_status {
    static bool attr_done[2][64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return MOCAP_ECUDA;
    const int which = head_dim == 128 ? 1 : 0;
    if (!attr_done[which][dev]) {
      if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               QkvLayout::kBytes) != cudaSuccess)
        return MOCAP_ECUDA;
      attr_done[which][dev] = true;
    }
    kern<<<grid, kThreads, QkvLayout::kBytes, reinterpret_cast<cudaStream_t>(stream)>>>(prm);
    return cudaGetLastError() == cudaSuccess ? MOCAP_OK : MOCAP_ECUDA;
  };
  return head_dim == 128 ? launch(qkv_rope_kernel<128>) : launch(qkv_rope_kernel<64>);
}
