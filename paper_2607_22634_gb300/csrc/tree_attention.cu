// presto_tree_attention: tree-masked GQA attention of the N tree tokens against the
// committed KV-cache prefix (target verification with a tree-structured attention
// mask, §5.1; App. C (I): each draft token sees the prefix and its ancestors).
//
// The GQA group of one kv head (G = Hq/Hkv query heads x N nodes = G*N rows) is a
// dense contraction against that head's keys, so it runs on the 5th-generation
// tensor cores, ping-ponging two 128-row tiles per CTA:
//   * one CTA per (sequence, kv head, pair of 128-row tiles, KV split);
//   * warp 16 issues TMA loads (both Q tiles once, then one K and one V tile of 128
//     keys at a time; K is refilled as soon as both QK^T products have read it, V as
//     soon as both PV products have);
//   * warp 17 issues tcgen05.mma into TMEM: S_t = Q_t K^T (128 fp32 columns per
//     tile) and O_t += P_t V (D columns per tile), interleaved so that the tensor
//     core works on one tile while the other tile's softmax runs;
//   * warps 0-7 and 8-15 run the softmax of tiles 0 and 1, two threads per query
//     row (TMEM lane), each on 64 of the 128 key columns: tcgen05.ld of S,
//     prefix-length and ancestor-bitmask masks, online softmax (the two halves of a
//     row exchange their maxima through shared memory), P (bf16, 128-byte swizzled
//     K-major) to shared memory.
//     The running maximum is only moved (and O rescaled in TMEM) when it grows by
//     more than 2^8, so most tiles skip the rescale;
//   * with several KV splits, the splits of one row block form a thread-block
//     cluster: each CTA leaves its fp32 O and (m, l) per row in its own shared
//     memory, the cluster synchronises, and each CTA merges a slice of the rows
//     from all peers through distributed shared memory (log-sum-exp weighting)
//     and writes them; no partials go to global memory.
// Every wait is bounded; on time-out the CTA records PRESTO_DEV_TIMEOUT and unwinds.
#include <cuda_bf16.h>

#include <cooperative_groups.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <initializer_list>
#include <mutex>

#include "common.cuh"

namespace presto {
namespace {

constexpr int kBM = 128;        // query rows per tile (TMEM lanes)
constexpr int kBN = 128;        // keys per tile
// 18 warps: per row tile 8 softmax warps (two threads per query row, each taking 64
// of the 128 key columns), then the TMA warp and the MMA warp
constexpr int kSoftWarps = 8;
constexpr int kThreads = (2 * kSoftWarps + 2) * 32;
constexpr int kTmaWarp = 2 * kSoftWarps;
constexpr int kMmaWarp = 2 * kSoftWarps + 1;
constexpr int kSoftThreads = kSoftWarps * 32;  // per tile
constexpr float kRescaleLog2 = 8.f;  // move the running max only when it grows by > 2^8
constexpr int kPanelBytes = 128 * 128;  // 128 rows x 128 bytes (64 bf16)
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr uint32_t kTmemCols = 512;  // S0 | S1 | O0 | O1, 128 columns each
// fp32 partial O rows left in shared memory for the cluster merge: padded so that
// a warp's 16-byte stores to 32 consecutive rows spread over the banks
template <int D>
constexpr int kPartStride = D + 4;
constexpr int kMaxSplits = 8;  // KV splits of a row block = CTAs of its (portable) cluster

struct Args {
  const int32_t* kv_len;
  const uint32_t* mask;
  const int32_t* n_nodes;
  int B, N, Hq, Hkv, G, Tmax, W, n_mt, tpc, n_groups, n_splits;  // tpc: row tiles per CTA
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  int32_t* dev_status;
};

template <int D>
struct Layout {
  static constexpr int kPanels = D / 64;
  static constexpr int kQBytes = kBM * D * 2;
  static constexpr int kTileBytes = kBN * D * 2;
  static constexpr int kPBytes = kBM * kBN * 2;
  static constexpr int kQ = 0;                       // Q of tile 0, then tile 1
  static constexpr int kK = kQ + 2 * kQBytes;
  static constexpr int kV = kK + kTileBytes;
  static constexpr int kP = kV + kTileBytes;         // P of tile 0, then tile 1
  static constexpr int kBytes = kP + 2 * kPBytes;
  static constexpr int kAlloc = kBytes + 1024;  // room to align the base to 1024
};

struct Bars {
  uint64_t q_full;
  uint64_t k_full, k_empty;
  uint64_t v_full, v_empty;
  uint64_t s_full[2], s_free[2];
  uint64_t p_full[2], o_done[2];
};

// Merge the KV splits of one row block (the CTAs of this cluster).  Every CTA holds
// the fp32 partial O (unnormalised) and (m, l) of its split for the block's rows in
// shared memory; CTA c of n merges rows [c*R/n, (c+1)*R/n) from all peers through
// distributed shared memory and writes the bf16 output and lse.  Phases: gather the
// peers' (m, l) of the slice, form per-row weights, then sum the peers' rows with
// all remote loads of an item issued together.
// Named barrier over `nthreads` threads that also returns the AND of `pred` over them.
__device__ __forceinline__ bool bar_and(int id, int nthreads, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n"
      " bar.red.and.pred q, %2, %3, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(pred)), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

template <int D>
__device__ void cluster_merge(const Args& a, int b, int g, int mt0, int ntiles, int nn,
                              uint8_t* smem, float2 (*part_ml)[kBM]) {
  namespace cg = cooperative_groups;
  cg::cluster_group cluster = cg::this_cluster();
  cluster.sync();  // every split's partial is in place
  const int nsp = static_cast<int>(cluster.num_blocks());
  const int me = static_cast<int>(cluster.block_rank());
  const int R = ntiles * kBM;
  const int r0 = me * R / nsp, r1 = (me + 1) * R / nsp, nr = r1 - r0;
  constexpr int kC4 = D / 4;  // float4 columns per row
  const int nodes_per_tile = kBM / a.G;
  // scratch after this CTA's own partial rows (the slice has <= kBM rows):
  // m then weight [row][split], l [row][split], 1/L [row], lse [row]
  float* wgt = reinterpret_cast<float*>(smem) + 2 * kBM * kPartStride<D>;
  float* lval = wgt + kBM * kMaxSplits;
  float* rinv = lval + kBM * kMaxSplits;
  float* rlse = rinv + kBM;
  for (int i = threadIdx.x; i < nr * nsp; i += kThreads) {
    const int row = r0 + i / nsp, s = i % nsp;
    const float2 ml = *cluster.map_shared_rank(&part_ml[row / kBM][row % kBM], s);
    wgt[(i / nsp) * kMaxSplits + s] = ml.x;
    lval[(i / nsp) * kMaxSplits + s] = ml.y;
  }
  __syncthreads();
  for (int i = threadIdx.x; i < nr; i += kThreads) {
    float* w = wgt + i * kMaxSplits;
    const float* lv = lval + i * kMaxSplits;
    float M = -INFINITY;
    for (int s = 0; s < nsp; ++s) M = fmaxf(M, w[s]);
    float L = 0.f;
    for (int s = 0; s < nsp; ++s) {
      const float ws = (M == -INFINITY || w[s] == -INFINITY) ? 0.f : ex2(w[s] - M);
      w[s] = ws;
      L += lv[s] * ws;
    }
    const int row = r0 + i;
    const int node = (mt0 + row / kBM) * nodes_per_tile + (row % kBM) / a.G;
    const bool used = node < nn && L > 0.f;
    rinv[i] = used ? 1.f / L : 0.f;
    rlse[i] = used ? (M + log2f(L)) * kLn2 : -INFINITY;
  }
  __syncthreads();
  for (int item = threadIdx.x; item < nr * kC4; item += kThreads) {
    const int i = item / kC4, c4 = item % kC4;
    const int rr = r0 + i;
    const int t = rr / kBM, r = rr % kBM;
    const int node = (mt0 + t) * nodes_per_tile + r / a.G, hh = r % a.G;
    if (node >= a.N) continue;
    const float* prow = reinterpret_cast<const float*>(smem) + rr * kPartStride<D> + c4 * 4;
    float4 o[kMaxSplits];
#pragma unroll
    for (int s = 0; s < kMaxSplits; ++s)
      if (s < nsp) o[s] = *reinterpret_cast<const float4*>(cluster.map_shared_rank(prow, s));
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int s = 0; s < kMaxSplits; ++s)
      if (s < nsp) {
        const float ws = wgt[i * kMaxSplits + s];
        acc.x += ws * o[s].x;
        acc.y += ws * o[s].y;
        acc.z += ws * o[s].z;
        acc.w += ws * o[s].w;
      }
    const float inv = rinv[i];
    const size_t orow = ((static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh) * D;
    const __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x * inv, acc.y * inv);
    const __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z * inv, acc.w * inv);
    uint2 u;
    u.x = *reinterpret_cast<const uint32_t*>(&lo);
    u.y = *reinterpret_cast<const uint32_t*>(&hi);
    *reinterpret_cast<uint2*>(a.out + orow + c4 * 4) = u;
    if (c4 == 0 && a.lse) a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh] = rlse[i];
  }
  cluster.sync();  // peers have finished reading this CTA's shared memory
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kc,
                const __grid_constant__ CUtensorMap tm_vc, const __grid_constant__ CUtensorMap tm_kt,
                const __grid_constant__ CUtensorMap tm_vt, const Args a) {
  using Ly = Layout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ Bars bars;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int idx = blockIdx.x;
  const int split = idx % a.n_splits;
  idx /= a.n_splits;
  const int mp = idx % a.n_groups;  // group of a.tpc row tiles
  idx /= a.n_groups;
  const int g = idx % a.Hkv;
  const int b = idx / a.Hkv;
  const int mt0 = mp * a.tpc;       // first row tile of the group
  const bool has1 = a.tpc == 2 && mt0 + 1 < a.n_mt;  // second tile present
  const int ntiles = has1 ? 2 : 1;

  int kv = a.kv_len[b];
  if (kv < 0 || kv > a.Tmax) {
    if (tid == 0) report(a.dev_status, PRESTO_DEV_BAD_KVLEN);
    kv = kv < 0 ? 0 : a.Tmax;
  }
  int nn = a.n_nodes[b];
  if (nn < 0 || nn > a.N) nn = nn < 0 ? 0 : a.N;
  const int prefix_tiles = (kv + kBN - 1) / kBN;
  const int per = (prefix_tiles + a.n_splits - 1) / a.n_splits;
  const int t_begin = min(split * per, prefix_tiles);
  const int n_prefix = min(prefix_tiles, t_begin + per) - t_begin;
  const int n_tree = split == a.n_splits - 1 ? (nn + kBN - 1) / kBN : 0;
  const int nt = n_prefix + n_tree;
  const int nodes_per_tile = kBM / a.G;

  __shared__ float2 part_ml[2][kBM];  // (m, l) per row of this CTA's split, log2 domain
  __shared__ float xchg[2][2][2][kBM];  // [iteration & 1][tile][half][row] row maxima
  __shared__ float lsum[2][2][kBM];     // [tile][half][row] row sums
  const bool clustered = a.n_splits > 1;
  if (nt == 0) {  // nothing to attend to in this split (CTA-uniform)
    if (tid < ntiles * kBM) {
      const int t = tid / kBM, r = tid % kBM;
      const int node = (mt0 + t) * nodes_per_tile + r / a.G, hh = r % a.G;
      if (clustered) {
        part_ml[t][r] = make_float2(-INFINITY, 0.f);
      } else if (node < a.N) {  // no keys at all: a zero row, lse -inf
        __nv_bfloat16* orow =
            a.out + ((static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh) * D;
        for (int c = 0; c < D; c += 8) *reinterpret_cast<uint4*>(orow + c) = make_uint4(0, 0, 0, 0);
        if (a.lse) a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh] = -INFINITY;
      }
    }
    if (clustered) cluster_merge<D>(a, b, g, mt0, ntiles, nn, smem, part_ml);
    return;
  }

  if (tid == 0) {
    mbar_init(&bars.q_full, 1);
    mbar_init(&bars.k_full, 1);
    mbar_init(&bars.k_empty, 1);
    mbar_init(&bars.v_full, 1);
    mbar_init(&bars.v_empty, 1);
    for (int t = 0; t < 2; ++t) {
      mbar_init(&bars.s_full[t], 1);
      mbar_init(&bars.s_free[t], kSoftThreads);
      mbar_init(&bars.p_full[t], kSoftThreads);
      mbar_init(&bars.o_done[t], 1);
    }
    abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  volatile int* abort = &abort_flag;
  auto fail = [&]() {
    *abort = 1;
    report(a.dev_status, PRESTO_DEV_TIMEOUT);
  };

  if (warp == kTmaWarp) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tensormap(&tm_q);
      prefetch_tensormap(&tm_kc);
      prefetch_tensormap(&tm_vc);
      prefetch_tensormap(&tm_kt);
      prefetch_tensormap(&tm_vt);
      mbar_arrive_expect_tx(&bars.q_full, ntiles * Ly::kQBytes);
      for (int t = 0; t < ntiles; ++t)
        for (int p = 0; p < Ly::kPanels; ++p)
          tma_load_3d(smem + Ly::kQ + t * Ly::kQBytes + p * kPanelBytes, &tm_q, p * 64, g * a.G,
                      b * a.N + (mt0 + t) * nodes_per_tile, &bars.q_full);
      auto load_kv = [&](int j, bool is_v) {
        uint64_t* bar = is_v ? &bars.v_full : &bars.k_full;
        uint8_t* dst = smem + (is_v ? Ly::kV : Ly::kK);
        mbar_arrive_expect_tx(bar, Ly::kTileBytes);
        for (int p = 0; p < Ly::kPanels; ++p) {
          if (j < n_prefix)
            tma_load_3d(dst + p * kPanelBytes, is_v ? &tm_vc : &tm_kc, p * 64,
                        (t_begin + j) * kBN, b * a.Hkv + g, bar);
          else
            tma_load_3d(dst + p * kPanelBytes, is_v ? &tm_vt : &tm_kt, p * 64, g,
                        b * a.N + (j - n_prefix) * kBN, bar);
        }
      };
      for (int j = 0; j < nt; ++j) {
        if (j > 0 && !mbar_wait(&bars.k_empty, (j - 1) & 1, abort)) {
          fail();
          break;
        }
        load_kv(j, false);
        if (j > 0 && !mbar_wait(&bars.v_empty, (j - 1) & 1, abort)) {
          fail();
          break;
        }
        load_kv(j, true);
      }
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(kBM, kBN, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, D, true);
      const uint32_t k_addr = smem_u32(smem + Ly::kK);
      const uint32_t v_addr = smem_u32(smem + Ly::kV);
      auto qk = [&](int t) {  // S_t = Q_t K^T
        const uint32_t q_addr = smem_u32(smem + Ly::kQ + t * Ly::kQBytes);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          mma_bf16(tmem_base + t * 128, smem_desc_sw128(q_addr + off, 16, 1024),
                   smem_desc_sw128(k_addr + off, 16, 1024), idesc_qk, kk > 0);
        }
        mma_commit(&bars.s_full[t]);
      };
      auto pv = [&](int t, bool acc) {  // O_t (+)= P_t V
        const uint32_t p_addr = smem_u32(smem + Ly::kP + t * Ly::kPBytes);
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk) {
          const uint32_t poff = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          const uint32_t voff = kk * 16 * 128;  // 16 keys x 128-byte rows
          mma_bf16(tmem_base + 256 + t * 128, smem_desc_sw128(p_addr + poff, 16, 1024),
                   smem_desc_sw128(v_addr + voff, kPanelBytes, 1024), idesc_pv,
                   (acc || kk > 0) ? 1u : 0u);
        }
        mma_commit(&bars.o_done[t]);
      };
      bool ok = mbar_wait(&bars.q_full, 0, abort) && mbar_wait(&bars.k_full, 0, abort);
      if (ok) {
        tc_fence_after();
        qk(0);
        if (has1) qk(1);
        mma_commit(&bars.k_empty);
      }
      for (int j = 0; ok && j < nt; ++j) {
        const bool next = j + 1 < nt;
        ok = mbar_wait(&bars.v_full, j & 1, abort) && mbar_wait(&bars.p_full[0], j & 1, abort);
        if (!ok) break;
        tc_fence_after();
        pv(0, j > 0);
        if (next) {
          ok = mbar_wait(&bars.k_full, (j + 1) & 1, abort) &&
               mbar_wait(&bars.s_free[0], j & 1, abort);
          if (!ok) break;
          tc_fence_after();
          qk(0);
        }
        if (has1) {
          ok = mbar_wait(&bars.p_full[1], j & 1, abort);
          if (!ok) break;
          tc_fence_after();
          pv(1, j > 0);
        }
        mma_commit(&bars.v_empty);
        if (next) {
          if (has1) {
            ok = mbar_wait(&bars.s_free[1], j & 1, abort);
            if (!ok) break;
            tc_fence_after();
            qk(1);
          }
          mma_commit(&bars.k_empty);
        }
      }
      if (!ok) fail();
    }
  } else if (warp < kSoftWarps * ntiles) {
    // ------------------------------------------------------------ softmax warps
    const int t = warp / kSoftWarps;           // row tile
    const int h = (warp % kSoftWarps) / 4;     // which 64 key columns / D/2 columns
    const int quad = warp & 3;                 // TMEM lane quadrant
    const int r = quad * 32 + lane;
    const uint32_t lane_addr = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t tS = tmem_base + t * 128 + h * 64 + lane_addr;
    const uint32_t tO = tmem_base + 256 + t * 128 + h * (D / 2) + lane_addr;
    uint8_t* sP = smem + Ly::kP + t * Ly::kPBytes + h * kPanelBytes;
    const int node = (mt0 + t) * nodes_per_tile + r / a.G;
    const int hh = r % a.G;
    const uint32_t* mrow =
        node < a.N ? a.mask + (static_cast<size_t>(b) * a.N + node) * a.W : nullptr;
    float m = -INFINITY, l = 0.f;  // m: running (possibly stale) max, log2 domain
    bool ok = true;
    for (int j = 0; j < nt; ++j) {
      // wait outcomes are made warp-uniform: tcgen05.ld needs the whole warp
      const bool got = __all_sync(0xffffffffu, ok && mbar_wait(&bars.s_full[t], j & 1, abort));
      uint32_t bits[2] = {0u, 0u};
      float mx = -INFINITY;
      if (got) {
        tc_fence_after();
        // masks: prefix keys beyond kv_len; tree keys outside the ancestor set
        if (j < n_prefix) {
          const int lim = kv - (t_begin + j) * kBN - h * 64;
          bits[0] = lim >= 32 ? 0xffffffffu : (lim <= 0 ? 0u : (1u << lim) - 1u);
          bits[1] = lim >= 64 ? 0xffffffffu : (lim <= 32 ? 0u : (1u << (lim - 32)) - 1u);
        } else {
          const int wi = (((j - n_prefix) * kBN) >> 5) + 2 * h;
          bits[0] = (mrow && wi < a.W) ? __ldg(mrow + wi) : 0u;
          bits[1] = (mrow && wi + 1 < a.W) ? __ldg(mrow + wi + 1) : 0u;
        }
        // pass 1: row max over this half's 64 columns, 32 at a time
#pragma unroll 1
        for (int c = 0; c < 2; ++c) {
          float v[32];
          tmem_ld32(tS + c * 32, v);
          const uint32_t bc = c ? bits[1] : bits[0];
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if ((bc >> e) & 1u) mx = fmaxf(mx, v[e] * a.scale_log2);
        }
      }
      // the two halves of each row meet here; a failed wait anywhere ends the loop
      // for both (barrier with an AND reduction)
      xchg[j & 1][t][h][r] = mx;
      if (!bar_and(1 + t, kSoftThreads, got)) {
        ok = false;
        break;
      }
      mx = fmaxf(mx, xchg[j & 1][t][1 - h][r]);
      // stale-max online softmax: move m only when the row max exceeds it by > 2^8
      const bool move = mx > m + kRescaleLog2;
      const float alpha = move ? ex2(m - mx) : 1.f;
      if (move) m = mx;
      const float m_use = m == -INFINITY ? 0.f : m;
      if (j > 0) {  // P buffer and O are free once PV_{j-1} of this tile completed
        if (!__all_sync(0xffffffffu, mbar_wait(&bars.o_done[t], (j - 1) & 1, abort))) {
          ok = false;  // leaves the loop at the next meeting point
          continue;
        }
        tc_fence_after();
      }
      // pass 2: P = exp2(S*scale - m) for this half's 64 keys of row r, into its
      // 64-key panel (bf16, 128-byte swizzle)
      float rs = 0.f;
#pragma unroll 1
      for (int c = 0; c < 2; ++c) {
        float v[32];
        tmem_ld32(tS + c * 32, v);
        const uint32_t bc = c ? bits[1] : bits[0];
        tmem_wait_ld();
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint4 u;
          uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int i0 = q * 8 + 2 * e;
            const float p0 = ((bc >> i0) & 1u) ? ex2(fmaf(v[i0], a.scale_log2, -m_use)) : 0.f;
            const float p1 =
                ((bc >> (i0 + 1)) & 1u) ? ex2(fmaf(v[i0 + 1], a.scale_log2, -m_use)) : 0.f;
            rs += p0 + p1;
            const __nv_bfloat162 pv2 = __floats2bfloat162_rn(p0, p1);
            w[e] = *reinterpret_cast<const uint32_t*>(&pv2);
          }
          const int chunk = c * 4 + q;
          *reinterpret_cast<uint4*>(sP + r * 128 + ((chunk ^ (r & 7)) << 4)) = u;
        }
      }
      tc_fence_before();
      mbar_arrive(&bars.s_free[t]);  // S_t may be overwritten by the next QK^T
      l = l * alpha + rs;
      if (j > 0 && __any_sync(0xffffffffu, move)) {
#pragma unroll
        for (int c = 0; c < D / 64; ++c) {
          float o[32];
          tmem_ld32(tO + c * 32, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] *= alpha;
          tmem_st32(tO + c * 32, o);
        }
        tmem_wait_st();
      }
      fence_proxy_async();  // make the P stores visible to the tensor core
      tc_fence_before();
      mbar_arrive(&bars.p_full[t]);
    }
    // row sum = the two halves' sums (same running max)
    lsum[t][h][r] = l;
    const bool all_ok = bar_and(1 + t, kSoftThreads, ok);
    l += lsum[t][1 - h][r];
    ok = __all_sync(0xffffffffu, all_ok && mbar_wait(&bars.o_done[t], (nt - 1) & 1, abort));
    if (ok) {
      tc_fence_after();
      // epilogue, this half's D/2 columns, 32 at a time: the normalised bf16 row, or
      // the fp32 partial left in this CTA's shared memory for the cluster merge.
      // (clustered) the partial overwrites Q/K/V/P space: tile 0's rows cover Q and
      // K, whose last readers (QK^T of both tiles) were issued before PV of tile 0
      // and are therefore complete once its last o_done arrived; tile 1's rows are
      // written after the last MMA of the CTA.  The other tile's P buffer lies
      // beyond both.
      const bool used = node < a.N && node < nn && l > 0.f;
      const float inv = used ? 1.f / l : 0.f;
      __nv_bfloat16* orow =
          a.out + ((static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh) * D + h * (D / 2);
      float* prow = reinterpret_cast<float*>(smem) + (t * kBM + r) * kPartStride<D> + h * (D / 2);
#pragma unroll 1
      for (int c = 0; c < D / 64; ++c) {
        float o[32];
        tmem_ld32(tO + c * 32, o);
        tmem_wait_ld();
        if (!clustered) {
          if (node < a.N) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              uint4 u;
              uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const __nv_bfloat162 o2 =
                    __floats2bfloat162_rn(o[q * 8 + 2 * e] * inv, o[q * 8 + 2 * e + 1] * inv);
                w[e] = *reinterpret_cast<const uint32_t*>(&o2);
              }
              *reinterpret_cast<uint4*>(orow + c * 32 + q * 8) = u;
            }
          }
        } else {
#pragma unroll
          for (int q = 0; q < 8; ++q)
            *reinterpret_cast<float4*>(prow + c * 32 + q * 4) =
                make_float4(o[q * 4], o[q * 4 + 1], o[q * 4 + 2], o[q * 4 + 3]);
        }
      }
      if (h == 0) {
        if (!clustered) {
          if (node < a.N && a.lse)
            a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh] =
                used ? (m + log2f(l)) * kLn2 : -INFINITY;
        } else {
          part_ml[t][r] = make_float2(m, l);
        }
      }
    } else {
      fail();
      if (clustered && h == 0) part_ml[t][r] = make_float2(-INFINITY, 0.f);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
  if (clustered) cluster_merge<D>(a, b, g, mt0, ntiles, nn, smem, part_ml);
}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}

// 3-D bf16 tensor map with a 128-byte-swizzled box (64 x b1 x b2 elements).
bool make_map(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
              uint64_t stride1_bytes, uint64_t stride2_bytes, uint32_t b1, uint32_t b2) {
  auto fn = encoder();
  if (!fn) return false;
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1_bytes, stride2_bytes};
  const cuuint32_t box[3] = {64, b1, b2};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct Plan {
  int G, n_mt, tpc, n_groups, n_splits;
  size_t ctas;
};


// active[s] = how many clusters of s CTAs (s = 1..kMaxSplits) can be resident on
// the GPU at once; 0 where that cluster size does not fit.
Plan make_plan(int B, int N, int Hq, int Hkv, int Tmax, const int* active) {
  Plan p;
  p.G = Hq / Hkv;
  p.n_mt = (N * p.G + kBM - 1) / kBM;
  const int prefix_tiles = (Tmax + kBN - 1) / kBN;
  int max_splits = prefix_tiles / 2 > 1 ? prefix_tiles / 2 : 1;
  if (max_splits > kMaxSplits) max_splits = kMaxSplits;
  // Choose row tiles per CTA (2 lets the softmax of one tile hide behind the
  // tensor-core work of the other) and the split count by the estimated time:
  // waves of resident clusters x (KV tiles per CTA x cost of one KV tile + fixed
  // cost), lightly penalising splits (each adds rows to merge).
  double best_cost = 1e30;
  p.tpc = 1;
  p.n_splits = 1;
  for (int tpc = 1; tpc <= 2; ++tpc) {
    const int groups = (p.n_mt + tpc - 1) / tpc;
    const long long units = static_cast<long long>(B) * Hkv * groups;
    const double tile_cost = tpc == 2 ? 1.15 : 1.0;
    for (int s = 1; s <= max_splits; ++s) {
      if (active[s] < 1) continue;
      const double waves = std::ceil(static_cast<double>(units) / active[s]);
      const double work = (prefix_tiles + 1.0) / s * tile_cost + 1.5;
      const double cost = waves * work * (1.0 + 0.02 * (s - 1));
      if (cost < best_cost - 1e-9) {
        best_cost = cost;
        p.tpc = tpc;
        p.n_splits = s;
      }
    }
  }
  p.n_groups = (p.n_mt + p.tpc - 1) / p.tpc;
  p.ctas = static_cast<size_t>(B) * Hkv * p.n_groups * p.n_splits;
  return p;
}

template <int D>
void set_smem_attr() {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         Layout<D>::kAlloc);
    cudaFuncSetAttribute(attn_kernel<D>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  });
}

// Resident-cluster counts for cluster sizes 1..kMaxSplits, for this kernel's block
// size and shared memory (queried once per device and D).
template <int D>
const int* active_clusters() {
  static int cached[64][kMaxSplits + 1];
  static bool done[64] = {false};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) dev = 0;
  std::lock_guard<std::mutex> lock(mu);
  int* act = cached[dev];
  if (done[dev]) return act;
  set_smem_attr<D>();
  act[0] = 0;
  for (int c = 1; c <= kMaxSplits; ++c) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(c);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = Layout<D>::kAlloc;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = c;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, attn_kernel<D>, &cfg) != cudaSuccess) {
      cudaGetLastError();
      n = 0;
    }
    act[c] = n;
  }
  if (act[1] < 1) act[1] = sm_count();  // a lone CTA always fits
  done[dev] = true;
  return act;
}

}  // namespace
}  // namespace presto

using namespace presto;

extern "C" size_t presto_attn_workspace(int B, int N, int Hq, int Hkv, int D, int Tmax) {
  if (B < 1 || N < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv || Tmax < 0 || (D != 64 && D != 128))
    return 0;
  // KV splits merge inside thread-block clusters; no device workspace is needed.
  return 256;
}

extern "C" int presto_tree_attention(const void* q, const void* k_cache, const void* v_cache,
                                     const int32_t* kv_len, int Tmax, const void* k_tree,
                                     const void* v_tree, const uint32_t* mask,
                                     const int32_t* n_nodes, int B, int N, int Hq, int Hkv, int D,
                                     float sm_scale, void* out, float* lse, void* ws,
                                     size_t ws_bytes, int32_t* dev_status,
                                     presto_stream_t stream) {
  PRESTO_CHECK_ARG(q && k_cache && v_cache && kv_len && k_tree && v_tree && mask && n_nodes && out);
  PRESTO_CHECK_ARG(B >= 1 && N >= 1 && Hq >= 1 && Hkv >= 1 && Tmax >= 1);
  PRESTO_CHECK_ARG(Hq % Hkv == 0);
  PRESTO_CHECK_ARG(sm_scale > 0.f && sm_scale < INFINITY);
  PRESTO_CHECK_LIMIT(D == 64 || D == 128);
  PRESTO_CHECK_LIMIT(N <= kMaxN);
  const int G = Hq / Hkv;
  PRESTO_CHECK_LIMIT(G <= kBM && (G & (G - 1)) == 0);
  for (const void* p : {q, k_cache, v_cache, k_tree, v_tree, static_cast<const void*>(out)})
    PRESTO_CHECK_ARG(reinterpret_cast<uintptr_t>(p) % 16 == 0);
  const int* active = D == 128 ? active_clusters<128>() : active_clusters<64>();
  const Plan p = make_plan(B, N, Hq, Hkv, Tmax, active);
  (void)ws;
  (void)ws_bytes;
  Args a{};
  const uint64_t e = 2;  // bf16 bytes
  CUtensorMap tq, tkc, tvc, tkt, tvt;
  const uint64_t Du = static_cast<uint64_t>(D);
  bool ok = make_map(&tq, q, Du, Hq, static_cast<uint64_t>(B) * N, Du * e, Du * Hq * e, G,
                     kBM / G) &&
            make_map(&tkc, k_cache, Du, Tmax, static_cast<uint64_t>(B) * Hkv, Du * e,
                     Du * Tmax * e, kBN, 1) &&
            make_map(&tvc, v_cache, Du, Tmax, static_cast<uint64_t>(B) * Hkv, Du * e,
                     Du * Tmax * e, kBN, 1) &&
            make_map(&tkt, k_tree, Du, Hkv, static_cast<uint64_t>(B) * N, Du * e, Du * Hkv * e, 1,
                     kBN) &&
            make_map(&tvt, v_tree, Du, Hkv, static_cast<uint64_t>(B) * N, Du * e, Du * Hkv * e, 1,
                     kBN);
  if (!ok) return PRESTO_ERR_CUDA;
  a.kv_len = kv_len;
  a.mask = mask;
  a.n_nodes = n_nodes;
  a.B = B;
  a.N = N;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = G;
  a.Tmax = Tmax;
  a.W = (N + 31) / 32;
  a.n_mt = p.n_mt;
  a.tpc = p.tpc;
  a.n_groups = p.n_groups;
  a.n_splits = p.n_splits;
  a.scale_log2 = sm_scale * kLog2e;
  a.out = static_cast<__nv_bfloat16*>(out);
  a.lse = lse;
  a.dev_status = dev_status;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(p.ctas));
  cfg.blockDim = dim3(kThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.n_splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t err;
  if (D == 128) {
    set_smem_attr<128>();
    cfg.dynamicSmemBytes = Layout<128>::kAlloc;
    err = cudaLaunchKernelEx(&cfg, attn_kernel<128>, tq, tkc, tvc, tkt, tvt, a);
  } else {
    set_smem_attr<64>();
    cfg.dynamicSmemBytes = Layout<64>::kAlloc;
    err = cudaLaunchKernelEx(&cfg, attn_kernel<64>, tq, tkc, tvc, tkt, tvt, a);
  }
  if (err != cudaSuccess) return PRESTO_ERR_CUDA;
  return launch_status();
}
