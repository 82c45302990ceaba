// attn_kernel.cuh -- the chunk attention kernel (device code) on sm_103a;
// chunk_attn.cu holds the host side (planning, launches, entry points).
//
// Sec. 2.2 / Eq. 1: chunk i's queries (global rows prefix .. prefix+len-1)
// attend to the KV of every earlier chunk plus a causal block over their own
// chunk; the attention work grows with the prefix, which is what LBCP
// balances.  The kernel computes, for query head h (KV head h / group) and
// global row t, O_t = softmax_{j<=t}(scale q_t.k_j) V and LSE_t = ln sum exp.
//
// Two forms.  CTA pairs (d = 128 with a multiple of four query heads per KV
// group, single and varlen launches; see control_roles_pair): two CTAs on
// two SMs share the KV group, row block and keys, each holds two heads, and
// tcgen05 cta_group::2 MMAs (M = 256) read K and V halves from both CTAs, so
// each SM stages and each SM's L2 traffic carries half of every K/V tile.
// The softmax warps and the layout of TMEM are the same in both forms.
// Single CTAs (every other shape) as follows.
//
// Design (one CTA = 128 query rows x up to two query heads of one KV group;
// CTAs are ordered KV-group-major, heaviest row block first within a group):
//   warp 0        TMA producer: Q tiles once, then K_j, V_j tiles (128 keys)
//                 through a 4-deep ring of 128-byte-swizzled smem stages.
//   warp 1        MMA issuer (one thread): S_s = Q_s K_j^T into TMEM, then
//                 O_s += P_s V_j with P_s read from TMEM; tcgen05.commit
//                 signals S ready / stage free / O final.  The next tile's
//                 K/V barriers are checked while a P V half is still queued,
//                 and V_j is released right after its last MMA, so no wait
//                 sits between the last MMA of a tile and the first of the
//                 next (a clock64 trace showed ~640 idle tensor cycles per
//                 tile there).
//   warps 4-7     softmax for head slot 0, warps 8-11 for slot 1 (a warp may
//                 touch only TMEM lanes 32*(warp%4) .. +31).  Thread r
//                 owns TMEM lane r = query row r, so row max / row sum are
//                 thread-local (no shuffles).  Online softmax in fp32, log2
//                 domain; O is rescaled in TMEM only when the running max grows
//                 by more than 2^8 (exact: the final 1/l uses the same max).
//                 P is written back to TMEM as packed bf16 (aliasing S), in
//                 two halves of 64 keys, each signalled on its own barrier
//                 so the first half of P V overlaps the second half's exps.
//   TMEM (512 columns): S0 [0,128) S1 [128,256) O0 [256,256+D) O1 [256+D, ..).
// The two slots share every K/V tile (two heads of one GQA group), so the
// tensor core alternates between them while the other slot's softmax runs.
// Key tiles entirely below the chunk's diagonal are unmasked; only the last
// one or two tiles apply the causal mask.  Rows and keys past the chunk end
// are zero-filled by TMA (the tensor maps end at prefix+len), so cache rows
// beyond the prefix are never read.
#pragma once

#include <cmath>
#include <cuda.h>
#include <cuda_bf16.h>

#include "internal.h"
#include "sm103_ptx.cuh"

namespace mocap {
namespace {


constexpr int kBlockM = 128;   // query rows per tile = TMEM lanes
constexpr int kBlockN = 128;   // keys per K/V tile
constexpr int kMaxSplits = 4;  // key-range splits of one chunk (split-KV)
constexpr int kThreads = 384;  // 3 warpgroups: {producer, MMA, 2 idle}, softmax 0, softmax 1
// Register split (setmaxnreg): the kernel is built for 168 registers per
// thread (384 x 168 = 64512 <= 65536); warpgroup 0 gives up to 56 and the two
// softmax warpgroups grow to 224: 128*56 + 256*224 = 64512.  The host refuses
// to launch if the compiled count differs, since an unbalanced split would
// block in setmaxnreg.inc.
constexpr int kLaunchRegs = 168;
constexpr uint32_t kRegsControl = 56;
constexpr uint32_t kRegsSoftmax = 224;
static_assert(kThreads * kLaunchRegs <= 65536, "register file");
static_assert(128 * kRegsControl + 256 * kRegsSoftmax <= kThreads * kLaunchRegs, "split");
constexpr int kBoxCols = 64;   // bf16 per 128-byte swizzled row
constexpr int kBoxBytes = kBlockM * kBoxCols * 2;  // 16 KB: one TMA box
constexpr uint32_t kTmemCols = 512;
constexpr float kMaxGrowthLog2 = 8.0f;  // rescale O only past a 2^8 max increase
constexpr uint64_t kDrainLimitNs = 20000000ull;  // 20 ms for in-flight copies

// One KV append carried by an attention launch (16-byte vectors): the K
// source's n_vec vectors go to k_cache + dst_vec, the V source's to
// v_cache + dst_vec.  `begin` is the segment's first index in the launch's
// flattened list of 2 * sum(n_vec) vectors, which the CTAs share out evenly.
struct AppendSeg {
  const uint4 *k_src;
  const uint4 *v_src;
  int64_t dst_vec;
  int64_t n_vec;
  int64_t begin;
};
constexpr int kMaxAppends = MOCAP_FUSED_APPEND_MAX;

struct ItemDesc {
  int64_t q_row;      // first packed Q/O row of the item
  int32_t prefix;     // keys before the chunk
  int32_t len;        // chunk rows
  int32_t q_blocks;   // ceil(len / 128)
  int32_t cta_begin;  // first CTA index of the item
};

template <int MAXI>
struct AttnParams {
  CUtensorMap tq[MAXI];  // Q  [len, Hq, D]           box {64, 1, 128}
  CUtensorMap tk[MAXI];  // K  [prefix+len, Hkv, D]   box {64, 1, 128} ({64, 1, 64}: CTA pairs)
  CUtensorMap tv[MAXI];  // V  [prefix+len, Hkv, D]   box {64, 1, 128}
  ItemDesc items[MAXI];
  __nv_bfloat16 *out;
  float *lse;
  uint32_t *status;
  int64_t lse_stride;
  int32_t n_items;
  int32_t n_q_heads;
  int32_t n_kv_heads;
  int32_t heads_per_group;
  int32_t pairs_per_group;
  float scale_log2;  // scale * log2(e)
  // Split-KV: when splits > 1 (single item only), CTA (unit, k) covers key
  // tiles [k n / splits, (k+1) n / splits) of its unit and writes fp32
  // partials instead of the final output: o_part [splits, len, Hq, D]
  // (normalised by its own row sum) and lse_part [splits, Hq, len].
  float *o_part;
  float *lse_part;
  int32_t splits;
  // KV appends done by this launch's otherwise idle warps 2-3 (cache rows no
  // CTA of the launch reads): n_app segments, app_total vectors in all.
  uint4 *k_cache_vec;
  uint4 *v_cache_vec;
  int64_t app_total;
  int32_t n_app;
  AppendSeg app[kMaxAppends];
  // Device item descriptors (DEV instantiations, items in device memory):
  // the item of every CTA, each item's ItemDesc and three tensor maps, and
  // the launch's CTA count, all written by the prepare kernel before the
  // launch (attn_varlen_dev.cuh).  CTAs at or past *dev_total exit at once.
  const ItemDesc *dev_items;
  const int32_t *dev_cta_item;
  const CUtensorMap *dev_maps;  // [item][Q, K, V]
  const int32_t *dev_total;
};

// Kernel parameters are limited to 32764 bytes (__grid_constant__ block).
static_assert(sizeof(AttnParams<MOCAP_VARLEN_MAX_ITEMS>) <= 32764, "kernel parameter space");

// Shared memory of one CTA.  Single-CTA form: two Q tiles and a ring of four
// stages, each holding one K or one V tile.  CTA-pair form (PAIR): each CTA
// stages only its half of every K tile (64 keys) and of every V tile (64
// dims), so a stage is half as large and the ring eight deep.
template <int D, bool PAIR = false>
struct Layout {
  static constexpr int kTileBytes = kBlockM * D * 2;  // one Q tile (one K or V tile)
  static constexpr int kStages = PAIR ? 8 : 4;
  static constexpr int kStageBytes = PAIR ? kTileBytes / 2 : kTileBytes;
  static constexpr int kQ = 0;                         // 2 Q tiles
  static constexpr int kRing = 2 * kTileBytes;
  static constexpr int kBars = kRing + kStages * kStageBytes;
  // barrier slots (8 bytes each)
  static constexpr int kBarQ = 0;
  static constexpr int kBarFull = 1;               // kStages
  static constexpr int kBarEmpty = 1 + kStages;    // kStages
  static constexpr int kBarS = 1 + 2 * kStages;    // 2
  static constexpr int kBarP = 3 + 2 * kStages;    // 2: keys 0..63 of P written
  static constexpr int kBarO = 5 + 2 * kStages;    // 2
  static constexpr int kBarDrain = 7 + 2 * kStages;
  static constexpr int kBarPHi = 8 + 2 * kStages;  // 2: keys 64..127 of P written
  static constexpr int kNumBars = 10 + 2 * kStages;
  static constexpr int kTmemSlot = kBars + 8 * kNumBars;
  static constexpr int kFlag = kTmemSlot + 4;
  // + slack for 1024-byte alignment; a CTA pair also keeps one K/V half of
  // slack past the barriers, so every MMA operand read stays inside this
  // CTA's allocation even if it reached past the last stage's half
  static constexpr int kBytes = kFlag + 4 + 1024 + (PAIR ? kStageBytes : 0);
};
static_assert(Layout<128>::kBytes <= 232448, "shared memory");
static_assert(Layout<128, true>::kBytes <= 232448, "shared memory");

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// S = Q K^T for one head slot: M=128, N=128, K=D; both operands K-major.
// q_desc / k_desc describe the tiles' first 16-column step; step kk starts
// (kk / 4) boxes and (kk % 4) * 32 bytes further (descriptor units of 16 B).
template <int D>
__device__ __forceinline__ void issue_qk(uint32_t s_tmem, uint64_t q_desc, uint64_t k_desc) {
  constexpr uint32_t idesc = idesc_bf16_f32(kBlockM, kBlockN, false, false);
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    const uint64_t off = static_cast<uint64_t>(((kk / 4) * kBoxBytes + (kk % 4) * 32) >> 4);
    mma_ss(s_tmem, q_desc + off, k_desc + off, idesc, kk > 0 ? 1u : 0u);
  }
}

// Half h of O += P V for one head slot: M=128, N=D, keys 64h .. 64h+63 (four
// K=16 steps).  P (A operand) lives in TMEM, 2 bf16 per column; V (B operand)
// is MN-major: d is contiguous, two 64-wide d halves 16 KB apart (leading byte
// offset), 8-key groups 1024 bytes apart (stride byte offset); step kk starts
// 16 keys = 2048 B further.
template <int D>
__device__ __forceinline__ void issue_pv_half(uint32_t o_tmem, uint32_t p_tmem, uint64_t v_desc,
                                              bool accumulate, int h) {
  constexpr uint32_t idesc = idesc_bf16_f32(kBlockM, D, false, true);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int kk = 4 * h + k;
    mma_ts(o_tmem, p_tmem + kk * 8, v_desc + static_cast<uint64_t>((kk * 2048) >> 4), idesc,
           (accumulate || k > 0) ? 1u : 0u);
  }
}

// One row of S (128 fp32 columns) into registers, with the causal mask
// applied when the tile crosses the diagonal (column c is key j*128 + c;
// `lim` is the last column this row may see).
__device__ __forceinline__ void load_scores(uint32_t taddr, bool masked, int lim, float (&x)[128]) {
  uint32_t r[128];
  tmem_ld128(taddr, r);
#pragma unroll
  for (int c = 0; c < 128; ++c) x[c] = __uint_as_float(r[c]);
  if (masked) {
#pragma unroll
    for (int c = 0; c < 128; ++c)
      if (c > lim) x[c] = -INFINITY;
  }
}

// Row max as 8 independent chains of 3-input max, then a short tree.
__device__ __forceinline__ float row_max(const float (&x)[128]) {
  float m[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) m[i] = fmax3(x[i], x[8 + i], x[16 + i]);
#pragma unroll
  for (int c = 24; c < 128; c += 16) {
#pragma unroll
    for (int i = 0; i < 8; ++i) m[i] = fmax3(m[i], x[c + i], c + 8 + i < 128 ? x[c + 8 + i] : m[i]);
  }
  const float a = fmax3(m[0], m[1], m[2]);
  const float b = fmax3(m[3], m[4], m[5]);
  return fmax3(a, b, fmaxf(m[6], m[7]));
}

__device__ __forceinline__ uint4 ld_stream_v4(const uint4 *ptr) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(ptr));
  return v;
}

// This CTA's share of the launch's KV appends: vectors [lo, hi) of the
// flattened list, lo = cta * total / ctas, copied by `nthreads` threads
// (tid 0 .. nthreads-1) with four 16-byte loads in flight per thread.  The
// destination rows are never read by this launch, so the copy needs no
// ordering with the attention work; kernel completion publishes it to later
// work on the stream.
// Kept out of line: inlined into the attention kernel it changed the
// register allocation of the whole kernel and cost about 12 % of its speed
// (out of line, about 1.4 %, measured on GB300).
template <int MAXI>
__device__ __noinline__ void append_share(const AttnParams<MAXI> &p, int tid, int nthreads) {
  if (p.n_app == 0) return;
  const int64_t ctas = gridDim.x;
  const int64_t cta = blockIdx.x;
  const int64_t lo = cta * p.app_total / ctas;
  const int64_t hi = (cta + 1) * p.app_total / ctas;
  constexpr int kInFlight = 4;
  for (int a = 0; a < p.n_app; ++a) {
    const AppendSeg &sg = p.app[a];
    const int64_t b = max(lo, sg.begin);
    const int64_t e = min(hi, sg.begin + 2 * sg.n_vec);
    for (int64_t i0 = b + tid; i0 < e; i0 += static_cast<int64_t>(kInFlight) * nthreads) {
      uint4 v[kInFlight];
#pragma unroll
      for (int u = 0; u < kInFlight; ++u) {
        const int64_t off = i0 + static_cast<int64_t>(u) * nthreads - sg.begin;
        if (off < e - sg.begin)
          v[u] = ld_stream_v4(off < sg.n_vec ? sg.k_src + off : sg.v_src + (off - sg.n_vec));
      }
#pragma unroll
      for (int u = 0; u < kInFlight; ++u) {
        const int64_t off = i0 + static_cast<int64_t>(u) * nthreads - sg.begin;
        if (off < e - sg.begin) {
          if (off < sg.n_vec) {
            p.k_cache_vec[sg.dst_vec + off] = v[u];
          } else {
            p.v_cache_vec[sg.dst_vec + (off - sg.n_vec)] = v[u];
          }
        }
      }
    }
  }
}

// Warpgroup 0: warp 0 is the TMA producer, warp 1 the MMA issuer (one lane
// each); warps 2-3 copy this CTA's share of the launch's KV appends, if any.
// The Q, K and V tensor maps of `item`: launch parameters, or (DEV) the maps
// a prepare kernel built in global memory, acquired for the tensormap proxy
// before their first use.
template <bool DEV, int MAXI>
__device__ __forceinline__ void item_maps(const AttnParams<MAXI> &p, int item,
                                          const CUtensorMap *&mq, const CUtensorMap *&mk,
                                          const CUtensorMap *&mv) {
  if constexpr (DEV) {
    mq = p.dev_maps + 3 * static_cast<int64_t>(item);
    mk = mq + 1;
    mv = mq + 2;
    tmap_acquire(mq);
    tmap_acquire(mk);
    tmap_acquire(mv);
  } else {
    mq = &p.tq[item];
    mk = &p.tk[item];
    mv = &p.tv[item];
  }
}

template <int D, int MAXI, bool APPEND, bool DEV = false>
__device__ __forceinline__ void control_roles(const AttnParams<MAXI> &p, uint32_t base,
                                              uint32_t bars, uint32_t tmem, uint32_t warp,
                                              uint32_t lane, int item, int g, int h0, int r0,
                                              int nslots, int t0, int n_kv) {
  using L = Layout<D>;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };
  if (warp == 0) {
    // ===================== TMA producer =====================================
    if (lane == 0) {
      const CUtensorMap *mq, *mk, *mv;
      item_maps<DEV>(p, item, mq, mk, mv);
      prefetch_tmap(mq);
      prefetch_tmap(mk);
      prefetch_tmap(mv);
      mbar_arrive_expect_tx(bar(L::kBarQ), nslots * L::kTileBytes);
      for (int s = 0; s < nslots; ++s)
        for (int c = 0; c < D / kBoxCols; ++c)
          tma_load_3d(base + L::kQ + s * L::kTileBytes + c * kBoxBytes, mq, bar(L::kBarQ),
                      c * kBoxCols, h0 + s, r0);
      const int n_seq = 2 * n_kv;  // K_0, V_0, K_1, V_1, ...
      bool ok = true;
      int seq = 0;
      for (; seq < n_seq; ++seq) {
        const int st = seq % L::kStages;
        if (seq >= L::kStages && !mbar_wait(bar(L::kBarEmpty + st), ((seq / L::kStages) - 1) & 1,
                                         p.status, kWaitLimitNs, true, kHintProducer)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(bar(L::kBarFull + st), L::kStageBytes);
        const CUtensorMap *m = (seq & 1) ? mv : mk;
        const int key0 = (t0 + (seq >> 1)) * kBlockN;
        for (int c = 0; c < D / kBoxCols; ++c)
          tma_load_3d(base + L::kRing + st * L::kStageBytes + c * kBoxBytes, m,
                      bar(L::kBarFull + st), c * kBoxCols, g, key0);
      }
      // Copies still in flight land before the CTA may exit.
      mbar_wait(bar(L::kBarQ), 0, p.status, kDrainLimitNs, false);
      for (int s2 = max(0, seq - L::kStages); s2 < seq; ++s2)
        mbar_wait(bar(L::kBarFull + s2 % L::kStages), (s2 / L::kStages) & 1, p.status, kDrainLimitNs,
                  false);
      // Normal exit: the last stage releases (tcgen05.commit arrivals) landed.
      if (ok)
        for (int s2 = max(0, n_seq - L::kStages); s2 < n_seq; ++s2)
          if (!mbar_wait(bar(L::kBarEmpty + s2 % L::kStages), (s2 / L::kStages) & 1, p.status)) break;
    }
  } else if (warp == 1) {
    // ===================== MMA issuer =======================================
    // The whole warp runs the loop (descriptors stay warp-uniform); one
    // elected lane issues the MMAs and their commits.
    const bool leader = elect_one();
    auto wait = [&](int b, int parity) {
      return mbar_wait_warp(bar(b), parity & 1, p.status, kHintMma);
    };
    // Descriptors of Q slot 0 and ring stage 0; other tiles are whole
    // multiples of kTileBytes further (descriptor start field in 16 B units).
    const uint64_t q_desc0 = sdesc_sw128(base + L::kQ, 16, 1024);
    const uint64_t k_desc0 = sdesc_sw128(base + L::kRing, 16, 1024);
    const uint64_t v_desc0 = sdesc_sw128(base + L::kRing, kBoxBytes, 1024);
    constexpr uint64_t kTileStep = static_cast<uint64_t>(L::kTileBytes >> 4);
    auto q_desc = [&](int s) { return q_desc0 + static_cast<uint64_t>(s) * kTileStep; };
    auto k_desc = [&](int st) { return k_desc0 + static_cast<uint64_t>(st) * kTileStep; };
    auto v_desc = [&](int st) { return v_desc0 + static_cast<uint64_t>(st) * kTileStep; };
    bool ok = wait(L::kBarQ, 0) && wait(L::kBarFull + 0, 0);
    if (ok) {
      tc_fence_after();
      if (leader) {
        for (int s = 0; s < nslots; ++s) {
          issue_qk<D>(tmem + s * kBlockN, q_desc(s), k_desc(0));
          tc_commit(bar(L::kBarS + s));
        }
        tc_commit(bar(L::kBarEmpty + 0));
      }
      __syncwarp();
      // tile 0's V and tile 1's K; later tiles' are checked one tile ahead,
      // while P V MMAs are still queued on the tensor core
      ok = wait(L::kBarFull + 1, 0);
      if (ok && n_kv > 1) ok = wait(L::kBarFull + 2 % L::kStages, 2 / L::kStages);
    }
    for (int j = 0; j < n_kv && ok; ++j) {
      const int sv = 2 * j + 1;  // V_j
      const int sk = 2 * j + 2;  // K_{j+1}
      const bool has_next = j + 1 < n_kv;
      for (int s = 0; s < nslots; ++s) {
        // P arrives in two halves (keys 0..63 on kBarP, 64..127 on kBarPHi),
        // each barrier completing once per tile.
        ok = wait(L::kBarP + s, j);
        if (!ok) break;
        tc_fence_after();
        if (leader)
          issue_pv_half<D>(tmem + 2 * kBlockN + s * D, tmem + s * kBlockN, v_desc(sv % L::kStages),
                           j > 0, 0);
        __syncwarp();
        if (s == nslots - 1 && has_next) {
          // V_{j+1} and K_{j+2}: waited here, with this P V half queued,
          // rather than at the next tile's start with the queue empty
          ok = wait(L::kBarFull + (sv + 2) % L::kStages, (sv + 2) / L::kStages);
          if (ok && j + 2 < n_kv) ok = wait(L::kBarFull + (sk + 2) % L::kStages, (sk + 2) / L::kStages);
          if (!ok) break;
        }
        ok = wait(L::kBarPHi + s, j);
        if (!ok) break;
        tc_fence_after();
        if (leader) {
          issue_pv_half<D>(tmem + 2 * kBlockN + s * D, tmem + s * kBlockN, v_desc(sv % L::kStages),
                           true, 1);
          if (s == nslots - 1) tc_commit(bar(L::kBarEmpty + sv % L::kStages));  // V_j read
          if (has_next) {
            issue_qk<D>(tmem + s * kBlockN, q_desc(s), k_desc(sk % L::kStages));
            tc_commit(bar(L::kBarS + s));
          } else {
            tc_commit(bar(L::kBarO + s));
          }
        }
        __syncwarp();
      }
      if (!ok) break;
      if (leader && has_next) tc_commit(bar(L::kBarEmpty + sk % L::kStages));  // K_{j+1} read
      __syncwarp();
    }
    // Every issued MMA completes before TMEM is released.
    if (leader) {
      tc_commit(bar(L::kBarDrain));
      mbar_wait(bar(L::kBarDrain), 0, p.status, kDrainLimitNs, false);
    }
    __syncwarp();
  } else if constexpr (APPEND) {
    append_share(p, static_cast<int>(threadIdx.x) - 64, 64);  // warps 2-3
  }
}

// CTA-pair control roles (d = 128, heads of a KV group taken four at a
// time: CTA r of the pair holds head slots {h0, h0 + 1} of its own head
// pair; both CTAs share the KV group, row block and key range).  Per key
// tile, CTA r stages keys 64 r .. 64 r + 63 of K and dims 64 r .. 64 r + 63
// of V; the first CTA's warp 1 issues cta_group::2 MMAs:
//   S_s = Q_s K^T   M = 256 (128 rows of each CTA's slot s), N = 128 keys
//   O_s += P_s V    M = 256 (P in each CTA's TMEM), N = 128 dims
// and its commits arrive on both CTAs' barriers.  Both CTAs' copies count on
// the first CTA's barriers, and so do both CTAs' P arrivals.
template <int MAXI, bool APPEND, bool DEV = false>
__device__ __forceinline__ void control_roles_pair(const AttnParams<MAXI> &p, uint32_t base,
                                                   uint32_t bars, uint32_t tmem, uint32_t warp,
                                                   uint32_t lane, uint32_t rank, int item, int g,
                                                   int h0, int r0, int nslots, int t0, int n_kv) {
  constexpr int D = 128;
  using L = Layout<D, true>;
  constexpr int S = L::kStages;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };
  const bool first = rank == 0;
  if (warp == 0) {
    // ===================== TMA producer (both CTAs) =========================
    if (lane == 0) {
      const CUtensorMap *mq, *mk, *mv;  // K in 64-row boxes: this CTA's half K tile
      item_maps<DEV>(p, item, mq, mk, mv);
      prefetch_tmap(mq);
      prefetch_tmap(mk);
      prefetch_tmap(mv);
      const uint32_t q_bar = cluster_addr(bar(L::kBarQ), 0);
      const uint32_t full0 = cluster_addr(bar(L::kBarFull), 0);
      if (first) mbar_arrive_expect_tx(bar(L::kBarQ), 2 * nslots * L::kTileBytes);
      for (int s = 0; s < nslots; ++s)
        for (int c = 0; c < D / kBoxCols; ++c)
          tma_load_3d_pair(base + L::kQ + s * L::kTileBytes + c * kBoxBytes, mq, q_bar,
                           c * kBoxCols, h0 + s, r0);
      const int n_seq = 2 * n_kv;  // K_0, V_0, K_1, V_1, ...
      bool ok = true;
      int seq = 0;
      for (; seq < n_seq; ++seq) {
        const int st = seq % S;
        if (seq >= S && !mbar_wait(bar(L::kBarEmpty + st), ((seq / S) - 1) & 1, p.status,
                                   kWaitLimitNs, true, kHintProducer)) {
          ok = false;
          break;
        }
        const uint32_t dst = base + L::kRing + st * L::kStageBytes;
        const int key0 = (t0 + (seq >> 1)) * kBlockN;
        if (first) mbar_arrive_expect_tx(bar(L::kBarFull + st), 2 * L::kStageBytes);
        if ((seq & 1) == 0) {  // K: this CTA's 64 keys, two 64-dim boxes of 8 KB
          for (int c = 0; c < D / kBoxCols; ++c)
            tma_load_3d_pair(dst + c * (kBoxBytes / 2), mk, full0 + 8u * st, c * kBoxCols, g,
                             key0 + 64 * static_cast<int>(rank));
        } else {  // V: this CTA's 64 dims of all 128 keys, one box of 16 KB
          tma_load_3d_pair(dst, mv, full0 + 8u * st, 64 * static_cast<int>(rank), g, key0);
        }
      }
      if (ok) {
        // the last stages' releases (commits after their MMAs) have arrived,
        // so every copy of this CTA has landed
        for (int s2 = max(0, n_seq - S); s2 < n_seq; ++s2)
          if (!mbar_wait(bar(L::kBarEmpty + s2 % S), (s2 / S) & 1, p.status)) break;
      } else if (first) {
        // copies still in flight (both CTAs' count here) land before exit
        mbar_wait(bar(L::kBarQ), 0, p.status, kDrainLimitNs, false);
        for (int s2 = max(0, seq - S); s2 < seq; ++s2)
          mbar_wait(bar(L::kBarFull + s2 % S), (s2 / S) & 1, p.status, kDrainLimitNs, false);
      }
    }
  } else if (warp == 1 && first) {
    // ===================== MMA issuer (first CTA) ===========================
    const bool leader = elect_one();
    auto wait = [&](int b, int parity) {
      return mbar_wait_warp(bar(b), parity & 1, p.status, kHintMma);
    };
    constexpr uint32_t idesc_s = idesc_bf16_f32(2 * kBlockM, kBlockN, false, false);
    constexpr uint32_t idesc_o = idesc_bf16_f32(2 * kBlockM, D, false, true);
    constexpr uint64_t kTileStep = static_cast<uint64_t>(L::kTileBytes >> 4);
    constexpr uint64_t kStageStep = static_cast<uint64_t>(L::kStageBytes >> 4);
    const uint64_t q_desc0 = sdesc_sw128(base + L::kQ, 16, 1024);
    const uint64_t k_desc0 = sdesc_sw128(base + L::kRing, 16, 1024);
    // V half: one 64-dim column of 128-byte atoms (no second column)
    const uint64_t v_desc0 = sdesc_sw128(base + L::kRing, kBoxBytes, 1024);
    // S_s = Q_s K^T: Q in 128-row boxes of 16 KB, the K half in 64-row boxes of 8 KB
    auto qk = [&](int s, int st) {
      const uint64_t qd = q_desc0 + static_cast<uint64_t>(s) * kTileStep;
      const uint64_t kd = k_desc0 + static_cast<uint64_t>(st) * kStageStep;
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint64_t qo = static_cast<uint64_t>(((kk / 4) * kBoxBytes + (kk % 4) * 32) >> 4);
        const uint64_t ko =
            static_cast<uint64_t>(((kk / 4) * (kBoxBytes / 2) + (kk % 4) * 32) >> 4);
        mma_pair(tmem + s * kBlockN, qd + qo, kd + ko, idesc_s, kk > 0 ? 1u : 0u);
      }
    };
    // half h of O_s += P_s V: keys 64h .. 64h+63 (four K=16 steps of 2 KB)
    auto pv_half = [&](int s, int st, bool accumulate, int h) {
      const uint64_t vd = v_desc0 + static_cast<uint64_t>(st) * kStageStep;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int kk = 4 * h + k;
        mma_ts_pair(tmem + 2 * kBlockN + s * D, tmem + s * kBlockN + kk * 8,
                    vd + static_cast<uint64_t>((kk * 2048) >> 4), idesc_o,
                    (accumulate || k > 0) ? 1u : 0u);
      }
    };
    bool ok = wait(L::kBarQ, 0) && wait(L::kBarFull + 0, 0);
    if (ok) {
      tc_fence_after();
      if (leader) {
        for (int s = 0; s < nslots; ++s) {
          qk(s, 0);
          commit_pair(bar(L::kBarS + s), 0x3);
        }
        commit_pair(bar(L::kBarEmpty + 0), 0x3);
      }
      __syncwarp();
      ok = wait(L::kBarFull + 1, 0);
      if (ok && n_kv > 1) ok = wait(L::kBarFull + 2 % S, 2 / S);
    }
    for (int j = 0; j < n_kv && ok; ++j) {
      const int sv = 2 * j + 1;  // V_j
      const int sk = 2 * j + 2;  // K_{j+1}
      const bool has_next = j + 1 < n_kv;
      for (int s = 0; s < nslots; ++s) {
        ok = wait(L::kBarP + s, j);  // both CTAs' keys 0..63 of P
        if (!ok) break;
        tc_fence_after();
        if (leader) pv_half(s, sv % S, j > 0, 0);
        __syncwarp();
        if (s == nslots - 1 && has_next) {  // V_{j+1}, K_{j+2} with this P V half queued
          ok = wait(L::kBarFull + (sv + 2) % S, (sv + 2) / S);
          if (ok && j + 2 < n_kv) ok = wait(L::kBarFull + (sk + 2) % S, (sk + 2) / S);
          if (!ok) break;
        }
        ok = wait(L::kBarPHi + s, j);
        if (!ok) break;
        tc_fence_after();
        if (leader) {
          pv_half(s, sv % S, true, 1);
          if (s == nslots - 1) commit_pair(bar(L::kBarEmpty + sv % S), 0x3);  // V_j read
          if (has_next) {
            qk(s, sk % S);
            commit_pair(bar(L::kBarS + s), 0x3);
          } else {
            commit_pair(bar(L::kBarO + s), 0x3);
          }
        }
        __syncwarp();
      }
      if (!ok) break;
      if (leader && has_next) commit_pair(bar(L::kBarEmpty + sk % S), 0x3);  // K_{j+1} read
      __syncwarp();
    }
    // Every issued MMA completes before TMEM is released.
    if (leader) {
      commit_pair(bar(L::kBarDrain), 0x1);
      mbar_wait(bar(L::kBarDrain), 0, p.status, kDrainLimitNs, false);
    }
    __syncwarp();
  } else if (warp >= 2) {
    if constexpr (APPEND) append_share(p, static_cast<int>(threadIdx.x) - 64, 64);  // warps 2-3
  }
}

// Warpgroups 1 and 2: online softmax for head slot (warp - 4) / 4, then the
// epilogue (O / l -> bf16, LSE).
template <int D, int MAXI, bool PAIR = false>
__device__ __forceinline__ void softmax_role(const AttnParams<MAXI> &p, uint32_t bars,
                                             uint32_t tmem, uint32_t warp, uint32_t lane,
                                             const ItemDesc &it, int h0, int r0, int nslots,
                                             int split, int t0, int n_kv, int qpos0,
                                             int n_unmasked) {
  using L = Layout<D, PAIR>;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };
  const int s = static_cast<int>(warp - 4) / 4;
  if (s < nslots) {
    // P-ready arrivals go to the barriers of the CTA that issues the MMAs:
    // this CTA, or the first CTA of a pair
    const uint32_t p_lo = PAIR ? cluster_addr(bar(L::kBarP + s), 0) : bar(L::kBarP + s);
    const uint32_t p_hi = PAIR ? cluster_addr(bar(L::kBarPHi + s), 0) : bar(L::kBarPHi + s);
    auto arrive_p = [&](uint32_t b) {
      if constexpr (PAIR) {
        mbar_arrive_cluster(b);
      } else {
        mbar_arrive(b);
      }
    };
    const uint32_t quarter = warp & 3u;
    const int row = static_cast<int>(quarter * 32 + lane);
    const uint32_t lane_addr = tmem + ((quarter * 32u) << 16);
    const uint32_t s_addr = lane_addr + s * kBlockN;
    const uint32_t o_addr = lane_addr + 2 * kBlockN + s * D;
    const int qpos = qpos0 + row;
    const float sl2 = p.scale_log2;
    float m = -INFINITY;  // running max of scale*log2(e)*s, possibly stale by < 2^8
    float l = 0.f;        // running sum of fp32 probabilities
    bool ok = true;
    for (int j = 0; j < n_kv; ++j) {
      if (!mbar_wait_warp(bar(L::kBarS + s), j & 1, p.status, kHintSoftmax)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float x[128];
      const int kt = t0 + j;  // key tile index
      const bool masked = kt >= n_unmasked;
      const int lim = qpos - kt * kBlockN;  // last visible column of this row
      load_scores(s_addr, masked, lim, x);
      const float mt = row_max(x) * sl2;
      if (j == 0) {
        m = mt;  // -inf only if this row sees no key of a split's first tile
      } else if (__any_sync(0xffffffffu, mt > m + kMaxGrowthLog2)) {
        // Rare: the running max grew by more than 2^8.  Rescale O and l,
        // then re-read S so its registers are free during the rescale.
        const float mn = fmaxf(m, mt);
        const float f = ex2_approx(m - mn);
        l *= f;
        m = mn;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(o_addr + c * 32, r);
#pragma unroll
          for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * f);
          tmem_st32(o_addr + c * 32, r);
        }
        tmem_st_wait();
        load_scores(s_addr, masked, lim, x);
      }
      // p = 2^(s * scale * log2 e - m): packed FMA for the argument, MUFU
      // for 2^x, packed adds into four independent partial sums.
      const uint64_t sl2x2 = f2(sl2, sl2);
      const float neg_m = m > -INFINITY ? -m : 0.0f;  // rows with no key yet: p = 0
      const uint64_t negm2 = f2(neg_m, neg_m);
      uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) {
        uint32_t pk[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int c = cc * 32 + 2 * e;
          float a, b;
          f2_split(ffma2(f2(x[c], x[c + 1]), sl2x2, negm2), a, b);
          a = ex2_approx(a);
          b = ex2_approx(b);
          acc[e & 3] = fadd2(acc[e & 3], f2(a, b));
          pk[e] = pack_bf16(a, b);
        }
        tmem_st16(s_addr + cc * 16, pk);  // P columns 16cc .. 16cc+15 alias S
        if (cc == 1) {  // keys 0..63 of P are in TMEM: the first half of P V may start
          tmem_st_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) arrive_p(p_lo);
        }
      }
      float sum0, sum1, sum2, sum3, sum4, sum5, sum6, sum7;
      f2_split(acc[0], sum0, sum1);
      f2_split(acc[1], sum2, sum3);
      f2_split(acc[2], sum4, sum5);
      f2_split(acc[3], sum6, sum7);
      sum0 = (sum0 + sum1) + (sum2 + sum3);
      sum1 = (sum4 + sum5) + (sum6 + sum7);
      l += sum0 + sum1;
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) arrive_p(p_hi);
    }
    if (ok) ok = mbar_wait_warp(bar(L::kBarO + s), 0, p.status);
    if (ok && p.splits > 1) {
      // Split-KV partial: O / l in fp32 and this range's natural-log LSE;
      // a row that saw no key in the range gets weight 0 (LSE = -inf).
      tc_fence_after();
      const bool valid = r0 + row < it.len;
      const bool any = l > 0.0f;
      const float inv = any ? 1.0f / l : 0.0f;
      const int64_t prow = static_cast<int64_t>(split) * it.len + r0 + row;
      float *dst = p.o_part + (prow * p.n_q_heads + h0 + s) * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(o_addr + c * 32, r);
        if (valid) {
          float4 *d4 = reinterpret_cast<float4 *>(dst + c * 32);
#pragma unroll
          for (int v = 0; v < 8; ++v)
            d4[v] = make_float4(__uint_as_float(r[4 * v]) * inv, __uint_as_float(r[4 * v + 1]) * inv,
                                __uint_as_float(r[4 * v + 2]) * inv,
                                __uint_as_float(r[4 * v + 3]) * inv);
        }
      }
      if (valid)
        p.lse_part[(static_cast<int64_t>(split) * p.n_q_heads + h0 + s) * it.len + r0 + row] =
            any ? (m + log2f(l)) * 0.69314718055994530942f : -INFINITY;
    } else if (ok) {
      tc_fence_after();
      const float inv = 1.0f / l;
      const bool valid = r0 + row < it.len;
      const int64_t orow = it.q_row + r0 + row;
      __nv_bfloat16 *dst = p.out + (orow * p.n_q_heads + h0 + s) * D;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(o_addr + c * 32, r);
        uint32_t pk[16];
#pragma unroll
        for (int e = 0; e < 16; ++e)
          pk[e] = pack_bf16(__uint_as_float(r[2 * e]) * inv, __uint_as_float(r[2 * e + 1]) * inv);
        if (valid) {
          uint4 *d4 = reinterpret_cast<uint4 *>(dst + c * 32);
#pragma unroll
          for (int v = 0; v < 4; ++v)
            d4[v] = make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
        }
      }
      if (valid)
        p.lse[static_cast<int64_t>(h0 + s) * p.lse_stride + orow] =
            (m + log2f(l)) * 0.69314718055994530942f;
    }
  }
}

// All 384 threads, reached from each warpgroup's own code path (the
// non-aligned barrier form allows different call sites).
__device__ __forceinline__ void cta_barrier() {
  asm volatile("barrier.sync 1, %0;" ::"n"(kThreads) : "memory");
}

// APPEND: the launch carries KV appends (warps 2-3 copy them).  A separate
// instantiation, so launches without appends run exactly the code they
// would without this feature.
// DEV: the items are device descriptors (the prepare kernel's tables).
template <int D, int MAXI, bool PAIR = false, bool APPEND = false, bool DEV = false>
__global__ void __launch_bounds__(kThreads, 1)
    chunk_attn_kernel(const __grid_constant__ AttnParams<MAXI> p) {
  using L = Layout<D, PAIR>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t *gbase = smem_raw + (base - raw);
  const uint32_t bars = base + L::kBars;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };
  volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(gbase + L::kTmemSlot);
  volatile uint32_t *flag = reinterpret_cast<volatile uint32_t *>(gbase + L::kFlag);

  const uint32_t warp = threadIdx.x >> 5;
  const uint32_t lane = threadIdx.x & 31u;

  // A launch after an expired wait does nothing (CTA-uniform decision; a
  // CTA pair takes its first CTA's reading after the set-up below, since
  // both CTAs must allocate TMEM together).
  if (threadIdx.x == 0) *flag = *reinterpret_cast<volatile uint32_t *>(p.status);
  __syncthreads();
  if (!PAIR && *flag != 0u) return;

  // ---- work item --------------------------------------------------------
  int item = 0;
  const int cta = static_cast<int>(blockIdx.x);
  if constexpr (DEV) {
    // the grid is an upper bound; a CTA pair's two CTAs exit together (the
    // count is a whole number of pairs)
    if (cta >= *p.dev_total) return;
    item = p.dev_cta_item[cta];
  } else {
    while (item + 1 < p.n_items && cta >= p.items[item + 1].cta_begin) ++item;
  }
  const ItemDesc it = DEV ? p.dev_items[item] : p.items[item];
  int w = cta - it.cta_begin;
  // CTA order: head pair fastest, then split, then row block (heaviest
  // first), then KV group slowest, so the CTAs resident at once mostly
  // stream the same group's K/V through L2 (less DRAM traffic and power).
  const int pair = w % p.pairs_per_group;
  w /= p.pairs_per_group;
  const int split = w % p.splits;
  w /= p.splits;
  const int qblock = it.q_blocks - 1 - w % it.q_blocks;
  const int g = w / it.q_blocks;
  const int r0 = qblock * kBlockM;
  const int h0 = g * p.heads_per_group + 2 * pair;
  const int nslots = min(2, p.heads_per_group - 2 * pair);
  const int qpos0 = it.prefix + r0;
  const int kv_len = it.prefix + it.len;
  const int kv_end = min(qpos0 + kBlockM, kv_len);
  const int n_tiles = (kv_end + kBlockN - 1) / kBlockN;
  const int n_unmasked = (qpos0 + 1) / kBlockN;  // tiles wholly at or below the diagonal
  // this CTA's key tiles: [t0, t0 + n_kv), split `split` of `splits`
  const int t0 = static_cast<int>(static_cast<int64_t>(split) * n_tiles / p.splits);
  const int n_kv =
      static_cast<int>(static_cast<int64_t>(split + 1) * n_tiles / p.splits) - t0;

  if (n_kv <= 0) {
    // No key tile in this split (the host never schedules one): an empty
    // partial, weight 0 in the combine, and this CTA's share of the appends.
    if constexpr (APPEND)
      if (warp == 2 || warp == 3) append_share(p, static_cast<int>(threadIdx.x) - 64, 64);
    if (p.splits > 1 && warp >= 4) {
      const int sl = static_cast<int>(warp - 4) / 4;
      const int row = static_cast<int>((warp & 3u) * 32 + lane);
      if (sl < nslots && r0 + row < it.len) {
        const int64_t prow = static_cast<int64_t>(split) * it.len + r0 + row;
        float *dst = p.o_part + (prow * p.n_q_heads + h0 + sl) * D;
        for (int c = 0; c < D; ++c) dst[c] = 0.0f;
        p.lse_part[(static_cast<int64_t>(split) * p.n_q_heads + h0 + sl) * it.len + r0 + row] =
            -INFINITY;
      }
    }
    return;
  }

  // ---- setup --------------------------------------------------------------
  if (warp == 1) {
    if constexpr (PAIR) {
      tmem_alloc_pair(base + L::kTmemSlot, kTmemCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(base + L::kTmemSlot, kTmemCols);
      tmem_relinquish();
    }
  }
  if (threadIdx.x == 0) {
    mbar_init(bar(L::kBarQ), 1);
    for (int s = 0; s < L::kStages; ++s) {
      mbar_init(bar(L::kBarFull + s), 1);
      mbar_init(bar(L::kBarEmpty + s), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(bar(L::kBarS + s), 1);
      mbar_init(bar(L::kBarP + s), PAIR ? 8 : 4);  // one arrive per softmax warp (both CTAs')
      mbar_init(bar(L::kBarO + s), 1);
    }
    mbar_init(bar(L::kBarDrain), 1);
    for (int s = 0; s < 2; ++s) mbar_init(bar(L::kBarPHi + s), PAIR ? 8 : 4);
    fence_mbar_init();
  }
  tc_fence_before();
  if constexpr (PAIR) {
    cluster_barrier();  // both CTAs' barriers exist before any copy, commit or remote arrive
  } else {
    __syncthreads();
  }
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if constexpr (PAIR) {
    const uint32_t rank = cta_rank_in_cluster();
    const bool run = ld_shared_cluster_u32(cluster_addr(smem_u32(const_cast<uint32_t *>(flag)), 0)) == 0u;
    if (run) {
      if (warp < 4) {
        setmaxnreg_dec<kRegsControl>();
        control_roles_pair<MAXI, APPEND, DEV>(p, base, bar(0), tmem, warp, lane, rank, item, g, h0, r0, nslots,
                                 t0, n_kv);
      } else {
        setmaxnreg_inc<kRegsSoftmax>();
        softmax_role<D, MAXI, true>(p, bar(0), tmem, warp, lane, it, h0, r0, nslots, split, t0,
                                    n_kv, qpos0, n_unmasked);
      }
    }
    tc_fence_before();
    cluster_barrier();  // MMAs drained, softmax and copies done in both CTAs
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc_pair(tmem, kTmemCols);
    }
    cluster_barrier();  // neither CTA leaves while the pair still shares state
  } else {
    if (warp < 4) {
      setmaxnreg_dec<kRegsControl>();
      control_roles<D, MAXI, APPEND, DEV>(p, base, bar(0), tmem, warp, lane, item, g, h0, r0, nslots, t0,
                             n_kv);
      tc_fence_before();
      cta_barrier();
      if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
      }
    } else {
      setmaxnreg_inc<kRegsSoftmax>();
      softmax_role<D, MAXI>(p, bar(0), tmem, warp, lane, it, h0, r0, nslots, split, t0, n_kv,
                            qpos0, n_unmasked);
      tc_fence_before();
      cta_barrier();
    }
  }
}

}  // namespace
}  // namespace mocap
