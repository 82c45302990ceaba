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
// Persistent warp-specialised tcgen05 GEMM on CTA pairs (clusters of two
// CTAs on two SMs, one pair per two SMs).  A pair computes a 256 x 256 output
// tile with cta_group::2 MMAs (M = 256, N = 256, K = 16): CTA r of the pair
// holds rows 128 r .. 128 r + 127 of the X tile and of the W tile in its
// shared memory, the tensor core reads both CTAs' halves, and each CTA's
// TMEM receives its own 128 rows x 256 columns.  Per K step a CTA stages
// 32 KB instead of the 48 KB of a single-CTA 128 x 256 tile, so the ring is
// deeper (6 stages) for the same shared memory, and L2 -> SM traffic per
// FLOP is two thirds of it.
//   warp 0      TMA producer (both CTAs): this CTA's X and W halves per K
//               step; completion is counted on the first CTA's barrier
//   warp 1      MMA issuer (first CTA only; converged warp, elected lane)
//               into one of two TMEM accumulators (2 x 256 columns); its
//               commits arrive on both CTAs' barriers
//   warps 2-5   epilogue (both CTAs): thread i owns TMEM lane i = its CTA's
//               output row i; fp32 -> RoPE (Q, K) -> bf16 -> 16-byte stores;
//               the second accumulator lets the next tile's main loop run
//               during this epilogue.
// Tiles are visited with the row tile fastest so pairs resident together
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

constexpr int kBM = 128;                      // rows per CTA (256 per pair tile)
constexpr int kBN = 256;                      // output features per tile
constexpr int kBK = 64;                       // hidden elements per K step
#ifndef MOCAP_QKV_STAGES
#define MOCAP_QKV_STAGES 6
#endif
constexpr int kStages = MOCAP_QKV_STAGES;
constexpr int kThreads = 192;                 // 6 warps
constexpr int kABytes = kBM * kBK * 2;        // 16 KB: this CTA's 128 rows of X
constexpr int kBBytes = (kBN / 2) * kBK * 2;  // 16 KB: this CTA's 128 rows of W
constexpr int kStageBytes = kABytes + kBBytes;
constexpr uint32_t kPairTx = 2u * kStageBytes;  // bytes landing per stage in the pair
constexpr int kMaxHalfDim = 64;               // d <= 128
constexpr uint16_t kBothCtas = 0x3;

struct QkvParams {
  CUtensorMap tx;  // X [len, hidden], box {64, 128}
  CUtensorMap tw;  // W [Nout, hidden], box {64, 128}
  __nv_bfloat16 *q_out;
  __nv_bfloat16 *k_cache;  // already offset to row `offset`
  __nv_bfloat16 *v_cache;
  uint32_t *status;
  int64_t pos0;            // position of row 0
  int32_t len, hidden, n_q_heads, n_kv_heads, head_dim;
  int32_t m_pairs, n_tiles, k_steps;
  uint64_t turn_step[kMaxHalfDim];  // theta^(-2j/d) / (2 pi) * 2^64, rounded down
};

struct QkvLayout {
  static constexpr int kRing = 0;
  static constexpr int kBars = kStages * kStageBytes;
  // full[S] (the first CTA's are used), empty[S], acc_full[2], acc_empty[2]
  // (the first CTA's: 4 local + 4 remote epilogue warps), drain
  static constexpr int kBarFull = 0, kBarEmpty = kStages, kBarAccFull = 2 * kStages,
                       kBarAccEmpty = 2 * kStages + 2, kBarDrain = 2 * kStages + 4,
                       kNumBars = 2 * kStages + 5;
  static constexpr int kTmemSlot = kBars + 8 * kNumBars;
  // Slack past the last stage as large as one W half: every operand read
  // of the MMA stays inside this CTA's allocation even if it reached past
  // the last stage's W half.
  static constexpr int kBytes = kTmemSlot + 8 + kBBytes + 1024;
};
static_assert(QkvLayout::kBytes <= 232448, "shared memory");

// Two 32-column loads of this warp's 32 lanes, one wait.
__device__ __forceinline__ void tmem_ld32x2(uint32_t ta, uint32_t tb, uint32_t (&a)[32],
                                            uint32_t (&b)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%64];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
      "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%65];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3]), "=r"(a[4]), "=r"(a[5]), "=r"(a[6]),
        "=r"(a[7]), "=r"(a[8]), "=r"(a[9]), "=r"(a[10]), "=r"(a[11]), "=r"(a[12]), "=r"(a[13]),
        "=r"(a[14]), "=r"(a[15]), "=r"(a[16]), "=r"(a[17]), "=r"(a[18]), "=r"(a[19]),
        "=r"(a[20]), "=r"(a[21]), "=r"(a[22]), "=r"(a[23]), "=r"(a[24]), "=r"(a[25]),
        "=r"(a[26]), "=r"(a[27]), "=r"(a[28]), "=r"(a[29]), "=r"(a[30]), "=r"(a[31]),
        "=r"(b[0]), "=r"(b[1]), "=r"(b[2]), "=r"(b[3]), "=r"(b[4]), "=r"(b[5]), "=r"(b[6]),
        "=r"(b[7]), "=r"(b[8]), "=r"(b[9]), "=r"(b[10]), "=r"(b[11]), "=r"(b[12]), "=r"(b[13]),
        "=r"(b[14]), "=r"(b[15]), "=r"(b[16]), "=r"(b[17]), "=r"(b[18]), "=r"(b[19]),
        "=r"(b[20]), "=r"(b[21]), "=r"(b[22]), "=r"(b[23]), "=r"(b[24]), "=r"(b[25]),
        "=r"(b[26]), "=r"(b[27]), "=r"(b[28]), "=r"(b[29]), "=r"(b[30]), "=r"(b[31])
      : "r"(ta), "r"(tb)
      : "memory");
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// Epilogue for one row of one 256-column tile: the tile's heads in order,
// each d columns; RoPE for Q and K heads (the angles of dims c .. c+31 are
// formed once per row and shared by the tile's heads), bf16, 16-byte
// stores.  `taddr` is this lane's TMEM address of the tile's first column.
template <int D>
__device__ __forceinline__ void emit_tile(const QkvParams &p, uint32_t taddr, int nt, int64_t row,
                                          bool valid, uint32_t pos) {
  constexpr int H = D / 2, kHeads = kBN / D;
  const int q_cols = p.n_q_heads * D, k_cols = p.n_kv_heads * D;
  const int col0 = nt * kBN;
  const bool any_rotate = col0 < q_cols + k_cols;  // heads run Q.., K.., V..
#pragma unroll
  for (int c = 0; c < H; c += 32) {
    float sn[32], cs[32];
    if (any_rotate) {
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        // top 32 bits of pos * step (mod 2^64): the fraction of a turn
        const uint64_t step = p.turn_step[c + e];
        const uint32_t turns =
            __umulhi(pos, static_cast<uint32_t>(step)) + pos * static_cast<uint32_t>(step >> 32);
        const float ang = static_cast<float>(static_cast<int32_t>(turns)) *
                          1.46291807926715968e-9f;  // 2 pi / 2^32
        __sincosf(ang, &sn[e], &cs[e]);
      }
    }
#pragma unroll 1
    for (int hs = 0; hs < kHeads; ++hs) {
      const int col = col0 + hs * D;  // first output feature of this head
      __nv_bfloat16 *dst;
      bool rotate = true;
      if (col < q_cols) {
        dst = p.q_out + (row * p.n_q_heads + col / D) * D;
      } else if (col < q_cols + k_cols) {
        dst = p.k_cache + (row * p.n_kv_heads + (col - q_cols) / D) * D;
      } else {
        dst = p.v_cache + (row * p.n_kv_heads + (col - q_cols - k_cols) / D) * D;
        rotate = false;
      }
      uint32_t lo[32], hi[32];
      tmem_ld32x2(taddr + hs * D + c, taddr + hs * D + H + c, lo, hi);  // dims c.., H+c..
      float a[32], b[32];
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        a[e] = __uint_as_float(lo[e]);
        b[e] = __uint_as_float(hi[e]);
      }
      if (rotate) {
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const float x0 = a[e], x1 = b[e];
          a[e] = x0 * cs[e] - x1 * sn[e];
          b[e] = x1 * cs[e] + x0 * sn[e];
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
}

template <int D>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    qkv_rope_kernel(const __grid_constant__ QkvParams p) {
  using L = QkvLayout;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;  // the same offset in both CTAs
  uint8_t *gbase = smem_raw + (base - raw);
  const uint32_t bars = base + L::kBars;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };
  volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(gbase + L::kTmemSlot);
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31u;
  const uint32_t rank = cta_rank_in_cluster();
  const bool first = rank == 0;
  const int pair = static_cast<int>(blockIdx.x >> 1), n_pairs = static_cast<int>(gridDim.x >> 1);

  __shared__ uint32_t abort_flag;
  if (threadIdx.x == 0) abort_flag = *reinterpret_cast<volatile uint32_t *>(p.status);
  if (warp == 1) {
    tmem_alloc_pair(base + L::kTmemSlot, 512);
    tmem_relinquish_pair();
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(bar(L::kBarFull + s), 1);
      mbar_init(bar(L::kBarEmpty + s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar(L::kBarAccFull + b), 1);
      mbar_init(bar(L::kBarAccEmpty + b), 8);  // 4 epilogue warps in each CTA
    }
    mbar_init(bar(L::kBarDrain), 1);
    fence_mbar_init();
  }
  tc_fence_before();
  cluster_barrier();  // both CTAs' barriers exist before any copy, commit or remote arrive
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int n_tiles_total = p.m_pairs * p.n_tiles;
  const bool run = abort_flag == 0u;

  if (warp == 0) {
    if (lane == 0 && run) {
      prefetch_tmap(&p.tx);
      prefetch_tmap(&p.tw);
      const uint32_t full0 = cluster_addr(bar(L::kBarFull), 0);  // the first CTA's full[0]
      int it = 0;  // global K-step counter across tiles (ring position)
      bool ok = true;
      for (int t = pair; t < n_tiles_total && ok; t += n_pairs) {
        const int mt = t % p.m_pairs, nt = t / p.m_pairs;
        const int row0 = mt * 2 * kBM + static_cast<int>(rank) * kBM;
        const int wrow0 = nt * kBN + static_cast<int>(rank) * (kBN / 2);
        for (int ks = 0; ks < p.k_steps; ++ks, ++it) {
          const int st = it % kStages;
          if (it >= kStages &&
              !mbar_wait(bar(L::kBarEmpty + st), ((it / kStages) - 1) & 1, p.status, kWaitLimitNs,
                         true, kHintProducer)) {
            ok = false;
            break;
          }
          const uint32_t sa = base + L::kRing + st * kStageBytes;
          if (first) mbar_arrive_expect_tx(bar(L::kBarFull + st), kPairTx);
          tma_load_2d_pair(sa, &p.tx, full0 + 8u * st, ks * kBK, row0);
          tma_load_2d_pair(sa + kABytes, &p.tw, full0 + 8u * st, ks * kBK, wrow0);
        }
      }
      // the MMAs that read the last stages have completed, so their copies landed
      if (ok)
        for (int s2 = max(0, it - kStages); s2 < it; ++s2)
          if (!mbar_wait(bar(L::kBarEmpty + s2 % kStages), (s2 / kStages) & 1, p.status)) break;
    }
  } else if (warp == 1) {
    if (first && run) {
      const bool leader = elect_one();
      constexpr uint32_t idesc = idesc_bf16_f32(2 * kBM, kBN, false, false);
      const uint64_t a0 = sdesc_sw128(base + L::kRing, 16, 1024);
      const uint64_t b0 = sdesc_sw128(base + L::kRing + kABytes, 16, 1024);
      constexpr uint64_t kStageStep = static_cast<uint64_t>(kStageBytes >> 4);
      int it = 0, tile_i = 0;
      bool ok = true;
      for (int t = pair; t < n_tiles_total && ok; t += n_pairs, ++tile_i) {
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
              mma_pair(acc, ad + 2 * kk, bd + 2 * kk, idesc, (ks > 0 || kk > 0) ? 1u : 0u);
            commit_pair(bar(L::kBarEmpty + st), kBothCtas);
          }
          __syncwarp();
        }
        if (!ok) break;
        if (leader) commit_pair(bar(L::kBarAccFull + buf), kBothCtas);
        __syncwarp();
      }
      if (leader) {  // every issued MMA completes before TMEM is released
        commit_pair(bar(L::kBarDrain), 0x1);
        mbar_wait(bar(L::kBarDrain), 0, p.status, 20000000ull, false);
      }
      __syncwarp();
    }
  } else if (run) {
    // epilogue warps 2..5: TMEM lane quarter = warp % 4
    const uint32_t quarter = warp & 3u;
    const int row_in_tile = static_cast<int>(quarter * 32 + lane);
    const uint32_t lane_addr = tmem + ((quarter * 32u) << 16);
    const uint32_t acc_empty0 = cluster_addr(bar(L::kBarAccEmpty), 0);  // the first CTA's
    int tile_i = 0;
    bool ok = true;
    for (int t = pair; t < n_tiles_total && ok; t += n_pairs, ++tile_i) {
      const int buf = tile_i & 1;
      const int use = tile_i >> 1;
      ok = mbar_wait_warp(bar(L::kBarAccFull + buf), use & 1, p.status, kHintSoftmax);
      if (!ok) break;
      tc_fence_after();
      const int mt = t % p.m_pairs, nt = t / p.m_pairs;
      const int row = mt * 2 * kBM + static_cast<int>(rank) * kBM + row_in_tile;
      emit_tile<D>(p, lane_addr + buf * kBN, nt, row, row < p.len,
                   static_cast<uint32_t>(p.pos0 + row));
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(acc_empty0 + 8u * buf);
    }
  }
  tc_fence_before();
  cluster_barrier();  // MMAs drained, epilogues and copies done in both CTAs
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, 512);
  }
  cluster_barrier();  // neither CTA leaves while the pair still shares state
}

// 2-D bf16 [rows, cols] row-major, box {64 cols, box_rows}, 128-byte swizzle.
bool make_map_2d(CUtensorMap *map, const void *ptr, int64_t rows, int64_t cols, int box_rows) {
  auto fn = tensor_map_encoder();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t elem[2] = {1u, 1u};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box,
            elem, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
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
  if (!make_map_2d(&prm.tx, x, len, hidden, kBM) ||
      !make_map_2d(&prm.tw, w_qkv, n_out, hidden, kBN / 2))
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
  prm.m_pairs = static_cast<int32_t>((len + 2 * kBM - 1) / (2 * kBM));
  prm.n_tiles = static_cast<int32_t>(n_out / kBN);
  prm.k_steps = (hidden + kBK - 1) / kBK;
  for (int j = 0; j < head_dim / 2; ++j) {
    const double turns = std::pow(static_cast<double>(rope_theta), -2.0 * j / head_dim) /
                         6.283185307179586477;  // < 1/(2 pi): fits below 2^62 once scaled
    prm.turn_step[j] = static_cast<uint64_t>(std::ldexp(turns, 64));
  }

  const int64_t tiles = static_cast<int64_t>(prm.m_pairs) * prm.n_tiles;
  const int grid = 2 * static_cast<int>(std::min<int64_t>(tiles, std::max(1, device_sm_count() / 2)));
  auto launch = [&](auto kern) -> mocap_status {
    // one flag set per kernel: both kernels have the same type, so this
    // lambda has one instantiation and indexes its flags by head_dim
    static ContextOnce once[2];
    ContextOnce &kern_once = once[head_dim == 128 ? 1 : 0];
    const uint64_t ctx = current_context();
    if (ctx == 0) return MOCAP_ECUDA;
    if (!kern_once.done(ctx)) {
      if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               QkvLayout::kBytes) != cudaSuccess)
        return MOCAP_ECUDA;
      kern_once.mark(ctx);
    }
    kern<<<grid, kThreads, QkvLayout::kBytes, reinterpret_cast<cudaStream_t>(stream)>>>(prm);
    return cudaGetLastError() == cudaSuccess ? MOCAP_OK : MOCAP_ECUDA;
  };
  return head_dim == 128 ? launch(qkv_rope_kernel<128>) : launch(qkv_rope_kernel<64>);
}
