// The long-run schedule of presto_tree_attention (tree-masked GQA attention of the
// N tree tokens against the committed KV-cache prefix, §5.1; App. C (I)), taken
// when each CTA walks many KV tiles: the entry points in tree_attention.cu choose
// it through pair_attn::run_tiles and launch it through pair_attn::launch.
//
// The GQA group of one kv head (G = Hq/Hkv query heads x N nodes = G*N rows) is a
// dense contraction against that head's keys, so it runs on the 5th-generation
// tensor cores, ping-ponging two 128-row tiles per CTA (over a long run the two
// tiles' softmax-to-tensor-core chains interleave, which beats a deeper S pipeline
// for one tile):
//   * one CTA per (sequence, kv head, pair of 128-row tiles, KV split);
//   * warp 8 loads both Q tiles, then K tiles of 128 keys into a ring; warp 10 loads
//     V tiles into another (TMA, 128-byte swizzle; 2 stages each at D = 128).  A K
//     slot is refilled once both QK^T products of its tile completed, a V slot once
//     both PV products did;
//   * warp 9 issues tcgen05.mma: S_t = Q_t K^T (128 fp32 TMEM columns per row tile)
//     and O_t += P_t V with P_t (bf16) read from TMEM, where the softmax wrote it over
//     S_t.  Per KV tile: PV(t0), QK^T(t0) of the next tile, PV(t1), QK^T(t1); each
//     QK^T waits for the completion of the PV that read the same TMEM, and the two
//     row tiles ping-pong so that one tile's softmax overlaps the other tile's
//     tensor work.  The whole warp runs the issue loop and one elected lane issues,
//     so descriptors stay on the uniform datapath;
//   * warps 0-3 and 4-7 run the softmax of tiles 0 and 1, one thread per query row
//     (TMEM lane): the row's 128 scores in registers (four tcgen05.ld in flight),
//     prefix-length and ancestor-bitmask masks (full prefix tiles skip them), online
//     softmax with packed fp32x2 arithmetic, P written back over S with tcgen05.st.
//     The running maximum is only moved (and O rescaled in TMEM) when it grows by
//     more than 2^8, so most tiles skip the rescale;
//   * with several KV splits (a row block's prefix and tree-key tiles dealt out in
//     equal runs), the splits of one row block form a thread-block cluster (up to 16
//     CTAs): each CTA writes its rows' fp32 (m, l) and O / l to the workspace (bf16
//     column quads, or float32 column pairs when the prefix is short; coalesced
//     either way), the cluster synchronises (release / acquire), and each CTA
//     merges a slice of the rows over the splits with log-sum-exp weights, all loads
//     of a row issued together.
// Every wait is bounded; on time-out the CTA records PRESTO_DEV_TIMEOUT, lets its
// copies and MMAs in flight complete (bounded), then frees its TMEM and exits.
#include <cuda_bf16.h>

#include <cooperative_groups.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <initializer_list>
#include <mutex>
#include <type_traits>

#include "attention_common.cuh"
#include "common.cuh"

namespace presto {
namespace {

using namespace attn;

// 11 warps: 0-3 and 4-7 run the softmax of row tiles 0 and 1 (one thread per query
// row = TMEM lane), 8 loads Q and K, 9 issues tensor-core MMAs, 10 loads V
constexpr int kThreads = 352;
constexpr int kKWarp = 8;
constexpr int kMmaWarp = 9;
constexpr int kVWarp = 10;
constexpr int kSoftThreads = 128;  // per tile
// TMEM columns: S of tile t (128 fp32) at 128t, overwritten in place by P of tile t
// (128 bf16 packed in pairs, its first 64 columns); O of tile t at 256 + 128t
constexpr uint32_t kTmemO = 256;

struct Args {
  const __nv_bfloat16* k_cache;  // [B, Hkv, Tmax, D] (for the L2 prefetch)
  const __nv_bfloat16* v_cache;
  const int32_t* kv_len;
  const uint32_t* mask;
  const int32_t* n_nodes;
  int B, N, Hq, Hkv, G, Tmax, W, n_mt, tpc, n_groups, n_splits;  // tpc: row tiles per CTA
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  float2* part_o;   // KV splits: O / l of each row, float32 [CTA][D / 2][2 * kBM] (column pairs)
  float2* part_ml;  // KV splits: (m, l) per row [CTA][2 * kBM], log2 domain
  int32_t* dev_status;
};

// Shared memory: Q of both row tiles, the K ring, the V ring.  Every operand is
// stored as 64-column panels of 128-byte rows with the 128-byte swizzle (128 rows
// per panel).  Ring depths: 2 at D = 128 (192 KB in all), 4 at D = 64.
template <int D>
struct Layout {
  static constexpr int kKStages = D == 64 ? 4 : 2;
  static constexpr int kVStages = D == 64 ? 4 : 2;
  static constexpr int kPanels = D / 64;
  static constexpr int kQPanel = kBM * kRowBytes;   // 16 KB
  static constexpr int kKVPanel = kBN * kRowBytes;  // 16 KB
  static constexpr int kQBytes = kBM * D * 2;
  static constexpr int kTileBytes = kBN * D * 2;    // one K or V tile
  static constexpr int kQ = 0;                          // tile 0, then tile 1
  static constexpr int kK = kQ + 2 * kQBytes;
  static constexpr int kV = kK + kKStages * kTileBytes;
  static constexpr int kBytes = kV + kVStages * kTileBytes;
  static constexpr int kAlloc = kBytes + 1024;  // room to align the base to 1024
};

constexpr int kMaxStages = 4;
struct Bars {
  uint64_t q_full;
  uint64_t k_full[kMaxStages], k_empty[kMaxStages];
  uint64_t v_full[kMaxStages], v_empty[kMaxStages];
  uint64_t s_full[2], p_full[2], o_done[2];
  uint64_t drain;  // after a timed-out wait: every MMA issued so far has completed
};


template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kc,
                const __grid_constant__ CUtensorMap tm_vc, const __grid_constant__ CUtensorMap tm_kt,
                const __grid_constant__ CUtensorMap tm_vt, const Args a) {
  namespace cg = cooperative_groups;
  using Ly = Layout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __shared__ Bars bars;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;
  __shared__ float mw[kBM][kMaxSplits + 1];  // split merge: per-row weights (slice <= kBM rows)
  __shared__ float mlse[kBM];                // split merge: per-row lse

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
  const bool clustered = a.n_splits > 1;
  const int nodes_per_tile = kBM / a.G;
  pdl_launch_dependents();

  if (tid == 0) {
    mbar_init(&bars.q_full, 1);
    for (int st = 0; st < kMaxStages; ++st) {
      mbar_init(&bars.k_full[st], 1);
      mbar_init(&bars.k_empty[st], 1);
      mbar_init(&bars.v_full[st], 1);
      mbar_init(&bars.v_empty[st], 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(&bars.s_full[t], 1);
      mbar_init(&bars.p_full[t], kSoftThreads);
      mbar_init(&bars.o_done[t], 1);
    }
    mbar_init(&bars.drain, 1);
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
  // before the dependency wait, ask L2 for this split's KV-prefix rows: no kernel of
  // the round writes the KV cache, and a prefetch is a hint that reads nothing into
  // the SM, so its DRAM traffic overlaps the previous kernels whatever they write.
  // The split's range is taken from kv_len as read now and the node budget N (the
  // exact split below uses the node count the build writes): a stale read only
  // misplaces the hint by a tile.
  if (tid == 0) {
    const int kvh = min(max(*reinterpret_cast<const volatile int32_t*>(a.kv_len + b), 0), a.Tmax);
    const int pt = (kvh + kBN - 1) / kBN;
    const int tot = pt + (a.N + kBN - 1) / kBN;
    const int per_h = (tot + a.n_splits - 1) / a.n_splits;
    const int tb = min(split * per_h, pt);
    const int te = min(tb + per_h, pt);
    if (te > tb) {
      const size_t row0 = (static_cast<size_t>(b) * a.Hkv + g) * a.Tmax;
      const int t0 = tb * kBN, t1 = min(te * kBN, kvh);
      const uint32_t bytes = static_cast<uint32_t>(t1 - t0) * D * 2u;
      prefetch_l2_bulk(a.k_cache + (row0 + t0) * D, bytes);
      prefetch_l2_bulk(a.v_cache + (row0 + t0) * D, bytes);
    }
  }
  pdl_wait();  // the mask and node counts come from the previous kernels on the stream
  const int kv_raw = ld_chain(a.kv_len + b);
  const int nn_raw = ld_chain(a.n_nodes + b);

  int kv = kv_raw;
  if (kv < 0 || kv > a.Tmax) {
    if (tid == 0) report(a.dev_status, PRESTO_DEV_BAD_KVLEN);
    kv = kv < 0 ? 0 : a.Tmax;
  }
  const int nn = nn_raw < 0 ? 0 : (nn_raw > a.N ? a.N : nn_raw);
  // split partials in float32 when the prefix is short: then a row averages few keys,
  // its values can be as large as single V entries, and the bf16 roundings of P, of a
  // bf16 partial and of the output could together reach 2e-2 of N(0, 1) values; with
  // a long prefix bf16 partials (half the merge traffic) lose nothing measurable
  const bool wide = kv < kWidePartialKeys;
  const int prefix_tiles = (kv + kBN - 1) / kBN;
  // the KV tiles of a row block, prefix tiles then tree tiles, in equal runs over the
  // splits: this split's local tile j is prefix tile t_begin + j for j < n_prefix,
  // else tree tile tree0 + (j - n_prefix)
  const int tree_tiles = (nn + kBN - 1) / kBN;
  const int total = prefix_tiles + tree_tiles;
  const int per = (total + a.n_splits - 1) / a.n_splits;
  const int t_begin = min(split * per, total);
  const int nt = min(total, t_begin + per) - t_begin;  // KV tiles of this split (CTA-uniform)
  const int n_prefix = max(0, min(nt, prefix_tiles - t_begin));
  const int tree0 = t_begin + n_prefix - prefix_tiles;

  volatile int* abort = &abort_flag;
  auto fail = [&]() {
    *abort = 1;
    report(a.dev_status, PRESTO_DEV_TIMEOUT);
  };

  int issued = 0;  // K or V tiles this warp's lane 0 has issued (the loaders)
  if (nt > 0 && warp == kKWarp) {
    // ------------------------------------------------------------ Q and K loads
    if (lane == 0) {
      prefetch_tensormap(&tm_q);
      prefetch_tensormap(&tm_kc);
      prefetch_tensormap(&tm_kt);
      mbar_arrive_expect_tx(&bars.q_full, ntiles * Ly::kQBytes);
      for (int t = 0; t < ntiles; ++t)
        for (int p = 0; p < Ly::kPanels; ++p)
          tma_load_3d(smem + Ly::kQ + t * Ly::kQBytes + p * Ly::kQPanel, &tm_q, p * 64, g * a.G,
                      b * a.N + (mt0 + t) * nodes_per_tile, &bars.q_full);
      // K_j -> slot j % Ly::kKStages, once both QK^T of K_{j - Ly::kKStages} completed
      for (int j = 0; j < nt; ++j) {
        const int st = j % Ly::kKStages;
        if (j >= Ly::kKStages && !mbar_wait(&bars.k_empty[st], (j / Ly::kKStages - 1) & 1, abort)) {
          fail();
          break;
        }
        uint8_t* dst = smem + Ly::kK + st * Ly::kTileBytes;
        mbar_arrive_expect_tx(&bars.k_full[st], Ly::kTileBytes);
        for (int p = 0; p < Ly::kPanels; ++p) {
          if (j < n_prefix)
            tma_load_3d(dst + p * Ly::kKVPanel, &tm_kc, p * 64, (t_begin + j) * kBN,
                        b * a.Hkv + g, &bars.k_full[st]);
          else
            tma_load_3d(dst + p * Ly::kKVPanel, &tm_kt, p * 64, g,
                        b * a.N + (tree0 + j - n_prefix) * kBN, &bars.k_full[st]);
        }
        issued = j + 1;
      }
    }
  } else if (nt > 0 && warp == kVWarp) {
    // ------------------------------------------------------------ V loads
    if (lane == 0) {
      prefetch_tensormap(&tm_vc);
      prefetch_tensormap(&tm_vt);
      // V_j -> slot j % Ly::kVStages, once both PV of V_{j - Ly::kVStages} completed
      for (int j = 0; j < nt; ++j) {
        const int st = j % Ly::kVStages;
        if (j >= Ly::kVStages && !mbar_wait(&bars.v_empty[st], (j / Ly::kVStages - 1) & 1, abort)) {
          fail();
          break;
        }
        uint8_t* dst = smem + Ly::kV + st * Ly::kTileBytes;
        mbar_arrive_expect_tx(&bars.v_full[st], Ly::kTileBytes);
        for (int p = 0; p < Ly::kPanels; ++p) {
          if (j < n_prefix)
            tma_load_3d(dst + p * Ly::kKVPanel, &tm_vc, p * 64, (t_begin + j) * kBN,
                        b * a.Hkv + g, &bars.v_full[st]);
          else
            tma_load_3d(dst + p * Ly::kKVPanel, &tm_vt, p * 64, g,
                        b * a.N + (tree0 + j - n_prefix) * kBN, &bars.v_full[st]);
        }
        issued = j + 1;
      }
    }
  } else if (nt > 0 && warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    // Per KV tile j and row tile t: PV_j(t) (P_t read from TMEM, where it overwrote
    // S_t), then QK_{j+1}(t) into the same TMEM, issued once PV_j(t) has completed
    // (its o_done), so S_t is never rewritten while P_t is still being read.  The whole warp runs this loop (wait outcomes made
    // warp-uniform); one elected lane issues each MMA and commit.
    constexpr uint32_t idesc_qk = idesc_bf16_f32(kBM, kBN, false);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, D, true);
    const uint64_t q_desc0 = smem_desc_sw128(smem_u32(smem + Ly::kQ), 16, 1024);
    const uint64_t k_desc0 = smem_desc_sw128(smem_u32(smem + Ly::kK), 16, 1024);
    const uint64_t v_desc0 = smem_desc_sw128(smem_u32(smem + Ly::kV), Ly::kKVPanel, 1024);
    auto wait = [&](uint64_t* bar, uint32_t parity) {
      const bool ok = __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
      if (ok) tc_fence_after();
      return ok;
    };
    // S_t = Q_t K_j^T
    auto qk = [&](int t, int j) {
      // descriptor start addresses are in 16-byte units in the low bits
      const uint64_t qd = q_desc0 + ((t * Ly::kQBytes) >> 4);
      const uint64_t kd = k_desc0 + (((j % Ly::kKStages) * Ly::kTileBytes) >> 4);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t qo = ((kk >> 2) * Ly::kQPanel + (kk & 3) * 32) >> 4;
        const uint32_t ko = ((kk >> 2) * Ly::kKVPanel + (kk & 3) * 32) >> 4;
        mma_bf16_warp(tmem_base + t * 128, qd + qo, kd + ko, idesc_qk, kk > 0);
      }
      mma_commit_warp(&bars.s_full[t]);
    };
    // O_t (+)= P_t V_j, P_t read from TMEM (8 columns = 16 keys per step)
    auto pv = [&](int t, int j) {
      if (!wait(&bars.p_full[t], j & 1)) return false;
      const uint64_t vd = v_desc0 + (((j % Ly::kVStages) * Ly::kTileBytes) >> 4);
#pragma unroll
      for (int kk = 0; kk < kBN / 16; ++kk)
        mma_bf16_ts_warp(tmem_base + kTmemO + t * 128, tmem_base + t * 128 + kk * 8,
                         vd + ((kk * 16 * kRowBytes) >> 4), idesc_pv, (j > 0 || kk > 0) ? 1u : 0u);
      mma_commit_warp(&bars.o_done[t]);
      return true;
    };
    bool ok = wait(&bars.q_full, 0) && wait(&bars.k_full[0], 0);
    if (ok) {
      qk(0, 0);
      if (has1) qk(1, 0);
      mma_commit_warp(&bars.k_empty[0]);
    }
    // ping-pong: tile 0's next S is issued right after its PV, so its softmax runs
    // while the tensor core works on tile 1, and the other way round
    for (int j = 0; ok && j < nt; ++j) {
      const int jn = j + 1;
      const bool more = jn < nt;
      ok = wait(&bars.v_full[j % Ly::kVStages], (j / Ly::kVStages) & 1) && pv(0, j);
      if (ok && more) {
        ok = wait(&bars.k_full[jn % Ly::kKStages], (jn / Ly::kKStages) & 1) &&
             wait(&bars.o_done[0], j & 1);
        if (ok) qk(0, jn);
      }
      if (ok && has1) {
        ok = pv(1, j);
        if (ok && more) {
          ok = wait(&bars.o_done[1], j & 1);
          if (ok) qk(1, jn);
        }
      }
      if (!ok) break;
      mma_commit_warp(&bars.v_empty[j % Ly::kVStages]);
      if (more) mma_commit_warp(&bars.k_empty[jn % Ly::kKStages]);
    }
    if (!ok && lane == 0) fail();
  } else if (nt > 0 && warp < 4 * ntiles) {
    // ------------------------------------------------------------ softmax warps
    const int t = warp >> 2;          // row tile
    const int quad = warp & 3;        // TMEM lane quadrant
    const int r = quad * 32 + lane;   // row of the tile
    const uint32_t lane_addr = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t tO = tmem_base + kTmemO + t * 128 + lane_addr;
    const uint32_t tS = tmem_base + t * 128 + lane_addr;  // S_t, then P_t in place
    const int node = (mt0 + t) * nodes_per_tile + r / a.G;
    const int hh = r % a.G;
    const uint32_t* mrow =
        node < a.N ? a.mask + (static_cast<size_t>(b) * a.N + node) * a.W : nullptr;
    float m = -INFINITY, l = 0.f;  // m: running (possibly stale) max, log2 domain
    bool ok = true;
    for (int j = 0; j < nt; ++j) {
      // wait outcomes are made warp-uniform: tcgen05.ld needs the whole warp.  S_j
      // ready also means PV_{j-1} of this tile completed (QK_j was issued after it),
      // so O_t may be rescaled and P_t rewritten.
      if (!__all_sync(0xffffffffu, mbar_wait(&bars.s_full[t], j & 1, abort))) {
        ok = false;
        break;
      }
      tc_fence_after();
      // masks of the four 32-key chunks: prefix keys beyond kv_len; tree keys outside
      // the ancestor set (a full prefix tile needs none)
      uint32_t bits[4];
      const bool full = j < n_prefix && kv - (t_begin + j) * kBN >= kBN;  // warp-uniform
      if (j < n_prefix) {
        const int lim = kv - (t_begin + j) * kBN;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int lc = lim - 32 * c;
          bits[c] = lc >= 32 ? 0xffffffffu : (lc <= 0 ? 0u : (1u << lc) - 1u);
        }
      } else {
        const int wi = ((tree0 + j - n_prefix) * kBN) >> 5;
#pragma unroll
        for (int c = 0; c < 4; ++c) bits[c] = (mrow && wi + c < a.W) ? ld_chain(mrow + wi + c) : 0u;
      }
      // the row's 128 scores: four loads in flight, one wait
      float v[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(tS + c * 32, *reinterpret_cast<float(*)[32]>(v + 32 * c));
      tmem_wait_ld();
      if (!full) {  // masked scores -> -inf (exp2 of -inf is 0)
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int e = 0; e < 32; ++e) v[32 * c + e] = ((bits[c] >> e) & 1u) ? v[32 * c + e] : -INFINITY;
      }
      float mx = fmaxf(fmaxf(row_max32(v), row_max32(v + 32)), fmaxf(row_max32(v + 64), row_max32(v + 96)));
      mx *= a.scale_log2;  // scale > 0 commutes with max
      // stale-max online softmax: move m only when the row max exceeds it by > 2^8
      const bool move = mx > m + kRescaleLog2;
      const float alpha = move ? ex2(m - mx) : 1.f;
      if (move) m = mx;
      const float m_use = m == -INFINITY ? 0.f : m;
      // p = exp2(s * scale - m), stored as bf16 pairs over the S columns (P covers the
      // first 64, all of S having been read); the row sum in packed chains
      const uint64_t sc2 = pack2(a.scale_log2, a.scale_log2), nm2 = pack2(-m_use, -m_use);
      uint64_t acc[2] = {0ull, 0ull};
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          float x0, x1;
          unpack2(fma2(pack2(v[32 * c + 2 * i], v[32 * c + 2 * i + 1]), sc2, nm2), x0, x1);
          const float p0 = ex2(x0), p1 = ex2(x1);
          acc[i & 1] = add2(acc[i & 1], pack2(p0, p1));
          const __nv_bfloat162 pv2 = __floats2bfloat162_rn(p0, p1);
          pk[i] = *reinterpret_cast<const uint32_t*>(&pv2);
        }
        tmem_st16(tS + c * 16, pk);
      }
      if (j > 0 && __any_sync(0xffffffffu, move)) {  // O_t *= alpha (rows that did not move: 1)
#pragma unroll 1
        for (int c = 0; c < D / 32; ++c) {
          float o[32];
          tmem_ld32(tO + c * 32, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] *= alpha;
          tmem_st32(tO + c * 32, o);
        }
      }
      float rs, rs1;
      unpack2(add2(acc[0], acc[1]), rs, rs1);
      l = l * alpha + (rs + rs1);
      tmem_wait_st();  // P (and a rescaled O) are in TMEM before the MMA is released
      tc_fence_before();
      mbar_arrive(&bars.p_full[t]);
    }
    if (ok)
      ok = __all_sync(0xffffffffu, mbar_wait(&bars.o_done[t], (nt - 1) & 1, abort));
    if (!ok) fail();
    if (clustered) {
      // this split's unnormalised row and (m, l) for the merge (a failed or empty
      // row is marked by m = -inf and contributes nothing)
      const size_t prow = static_cast<size_t>(blockIdx.x) * 2 * kBM + t * kBM + r;
      a.part_ml[prow] = ok ? make_float2(m, l) : make_float2(-INFINITY, 0.f);
      if (ok) {
        tc_fence_after();
        // the row normalised by its own l (values stay within the range of V), laid
        // out so that a warp's 32 rows of one column group are 256 contiguous bytes:
        // bf16 column quads, or float32 column pairs when the sequence's prefix is
        // short (wide_partials)
        const float inv = l > 0.f ? 1.f / l : 0.f;
        if (wide) {
          float2* dst = reinterpret_cast<float2*>(a.part_o) +
                        static_cast<size_t>(blockIdx.x) * (D / 2) * 2 * kBM + t * kBM + r;
#pragma unroll 1
          for (int c = 0; c < D / 32; ++c) {
            float o[32];
            tmem_ld32(tO + c * 32, o);
            tmem_wait_ld();
#pragma unroll
            for (int q = 0; q < 16; ++q)
              dst[(c * 16 + q) * 2 * kBM] = make_float2(o[q * 2] * inv, o[q * 2 + 1] * inv);
          }
        } else {
          uint2* dst = reinterpret_cast<uint2*>(a.part_o) +
                       static_cast<size_t>(blockIdx.x) * (D / 4) * 2 * kBM + t * kBM + r;
#pragma unroll 1
          for (int c = 0; c < D / 32; ++c) {
            float o[32];
            tmem_ld32(tO + c * 32, o);
            tmem_wait_ld();
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const __nv_bfloat162 lo = __floats2bfloat162_rn(o[q * 4] * inv, o[q * 4 + 1] * inv);
              const __nv_bfloat162 hi = __floats2bfloat162_rn(o[q * 4 + 2] * inv, o[q * 4 + 3] * inv);
              dst[(c * 8 + q) * 2 * kBM] = make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                                                      *reinterpret_cast<const uint32_t*>(&hi));
            }
          }
        }
      }
    } else if (ok) {
      tc_fence_after();
      // the normalised bf16 row, 32 columns at a time, and its lse
      const bool used = node < a.N && node < nn && l > 0.f;
      const float inv = used ? 1.f / l : 0.f;
      __nv_bfloat16* orow =
          a.out + ((static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh) * D;
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        float o[32];
        tmem_ld32(tO + c * 32, o);
        tmem_wait_ld();
        if (node < a.N) {
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint4 w4;
            uint32_t* w = reinterpret_cast<uint32_t*>(&w4);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const __nv_bfloat162 o2 =
                  __floats2bfloat162_rn(o[q * 8 + 2 * e] * inv, o[q * 8 + 2 * e + 1] * inv);
              w[e] = *reinterpret_cast<const uint32_t*>(&o2);
            }
            *reinterpret_cast<uint4*>(orow + c * 32 + q * 8) = w4;
          }
        }
      }
      if (node < a.N && a.lse)
        a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh] =
            used ? (m + log2f(l)) * kLn2 : -INFINITY;
    }
  }

  // ---- unwind after a timed-out wait.  Before the TMEM is freed and the CTA exits,
  // nothing asynchronous may still target them: each loader waits (bounded) for the
  // last copy it issued into every stage (and for Q), whether or not anyone consumed
  // it, and the MMA warp commits to the drain barrier, which completes once every
  // MMA it issued has.  A drain wait that gives up too means the GPU no longer
  // answers; the status word already holds PRESTO_DEV_TIMEOUT.
  if (__syncthreads_or(*abort)) {
    if (nt > 0 && (warp == kKWarp || warp == kVWarp) && lane == 0) {
      uint64_t* full = warp == kKWarp ? bars.k_full : bars.v_full;
      const int S = warp == kKWarp ? Ly::kKStages : Ly::kVStages;
      if (warp == kKWarp) mbar_wait(&bars.q_full, 0, nullptr);
      for (int j = max(0, issued - S); j < issued; ++j) mbar_wait(&full[j % S], (j / S) & 1, nullptr);
    }
    if (nt > 0 && warp == kMmaWarp) {
      mma_commit_warp(&bars.drain);
      mbar_wait(&bars.drain, 0, nullptr);
    }
  }

  if (!clustered) {
    if (nt == 0 && tid < ntiles * kBM) {  // no keys at all: a zero row, lse -inf
      const int t = tid / kBM, r = tid % kBM;
      const int node = (mt0 + t) * nodes_per_tile + r / a.G, hh = r % a.G;
      if (node < a.N) {
        __nv_bfloat16* orow =
            a.out + ((static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh) * D;
        for (int c = 0; c < D; c += 8) *reinterpret_cast<uint4*>(orow + c) = make_uint4(0, 0, 0, 0);
        if (a.lse) a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh] = -INFINITY;
      }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
      tc_fence_after();
      tmem_dealloc(tmem_base, kTmemCols);
    }
    return;
  }

  // ---------------------------------------------------------------- split merge
  // The KV splits of this row block are the CTAs of the cluster; each has left its
  // rows' (m, l) and unnormalised O in the workspace.  Rows are dealt out in slices,
  // one per CTA, and each CTA combines its slice over the splits with log-sum-exp
  // weights (the partials stay in L2).
  if (nt == 0 && tid < ntiles * kBM)  // an empty split contributes nothing
    a.part_ml[static_cast<size_t>(blockIdx.x) * 2 * kBM + tid] = make_float2(-INFINITY, 0.f);
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
  // release / acquire at cluster scope: every split's partial rows are visible
  cg::this_cluster().sync();
  const int R = ntiles * kBM;
  const int nsp = a.n_splits;
  const int slice = (R + nsp - 1) / nsp;
  const size_t cta0 = static_cast<size_t>(blockIdx.x - split);  // first CTA of the cluster
  const int r0 = split * slice;
  const int nr = max(0, min(R, r0 + slice) - r0);
  // One item = one row of the slice x one column group (a bf16 quad or a float32
  // pair), rows fastest (coalesced partial loads).  Each thread's first item is
  // loaded before the per-row weights are formed (one thread per row, into shared
  // memory), so the usual case costs one L2 round trip.
  auto merge = [&](auto wide_tag) {
    constexpr bool kWide = decltype(wide_tag)::value;
    using PT = std::conditional_t<kWide, float2, uint2>;
    constexpr int kCG = kWide ? D / 2 : D / 4;  // column groups per row
    const PT* part = reinterpret_cast<const PT*>(a.part_o);
    const int nitems = nr * kCG;
    auto load_item = [&](int item, PT (&o)[kMaxSplits]) {
      const int cg = item / max(nr, 1), row = r0 + item % max(nr, 1);
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s)
        o[s] = (item < nitems && s < nsp) ? __ldcg(part + ((cta0 + s) * kCG + cg) * 2 * kBM + row)
                                         : PT{};
    };
    PT oa[kMaxSplits];
    load_item(tid, oa);
    if (tid < nr) {
      // the row's weights over the splits, w_s l_s / L (a split without keys for the
      // row has m = -inf and weight 0), and its lse
      const int row = r0 + tid;
      float2 ml[kMaxSplits];
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s)
        ml[s] = s < nsp ? __ldcg(a.part_ml + (cta0 + s) * 2 * kBM + row) : make_float2(-INFINITY, 0.f);
      float M = -INFINITY;
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s) M = fmaxf(M, ml[s].x);
      float L = 0.f;
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s) {
        const float wl = (M == -INFINITY || ml[s].x == -INFINITY) ? 0.f : ex2(ml[s].x - M) * ml[s].y;
        mw[tid][s] = wl;
        L += wl;
      }
      const int node = (mt0 + row / kBM) * nodes_per_tile + (row % kBM) / a.G;
      const bool used = node < nn && L > 0.f;
      const float inv = used ? 1.f / L : 0.f;
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s) mw[tid][s] *= inv;
      mlse[tid] = used ? (M + log2f(L)) * kLn2 : -INFINITY;
    }
    __syncthreads();
    auto finish_item = [&](int item, const PT (&o)[kMaxSplits]) {
      if (item >= nitems) return;
      const int cg = item / nr, i = item % nr;
      const int row = r0 + i;
      const int node = (mt0 + row / kBM) * nodes_per_tile + (row % kBM) / a.G;
      const int hh = (row % kBM) % a.G;
      if (node >= a.N) return;
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s) {
        // weight 0: an absent split, or one without keys for this row (an empty
        // split writes no partial O, so its workspace bytes are whatever is there)
        const float w = mw[i][s];
        if (w != 0.f) {
          if constexpr (kWide) {
            acc[0] = fmaf(w, o[s].x, acc[0]);
            acc[1] = fmaf(w, o[s].y, acc[1]);
          } else {
            acc[0] = fmaf(w, __uint_as_float(o[s].x << 16), acc[0]);
            acc[1] = fmaf(w, __uint_as_float(o[s].x & 0xffff0000u), acc[1]);
            acc[2] = fmaf(w, __uint_as_float(o[s].y << 16), acc[2]);
            acc[3] = fmaf(w, __uint_as_float(o[s].y & 0xffff0000u), acc[3]);
          }
        }
      }
      const size_t orow = ((static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh) * D;
      const __nv_bfloat162 lo = __floats2bfloat162_rn(acc[0], acc[1]);
      if constexpr (kWide) {
        *reinterpret_cast<__nv_bfloat162*>(a.out + orow + cg * 2) = lo;
      } else {
        const __nv_bfloat162 hi = __floats2bfloat162_rn(acc[2], acc[3]);
        *reinterpret_cast<uint2*>(a.out + orow + cg * 4) =
            make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi));
      }
      if (cg == 0 && a.lse) a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh] = mlse[i];
    };
    finish_item(tid, oa);
    for (int item = tid + kThreads; item < nitems; item += kThreads) {
      load_item(item, oa);
      finish_item(item, oa);
    }
  };
  if (wide)
    merge(std::true_type{});
  else
    merge(std::false_type{});
}

// ------------------------------------------------------------------ host side

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
  const int tree_tiles = (N + kBN - 1) / kBN;
  int max_splits = (prefix_tiles + tree_tiles) / 2 > 1 ? (prefix_tiles + tree_tiles) / 2 : 1;
  if (max_splits > kMaxSplits) max_splits = kMaxSplits;
  // Choose row tiles per CTA (2 lets the softmax of one tile hide behind the
  // tensor-core work of the other, and reads K/V once for both) and the split
  // count by the estimated time: waves of resident clusters x (KV tiles per CTA x
  // cost of one KV tile + fixed cost), lightly penalising splits (each adds rows
  // to merge).
  double best_cost = 1e30;
  p.tpc = 1;
  p.n_splits = 1;
  for (int tpc = 1; tpc <= 2; ++tpc) {
    const int groups = (p.n_mt + tpc - 1) / tpc;
    const long long units = static_cast<long long>(B) * Hkv * groups;
    const double tile_cost = tpc == 2 ? 1.3 : 1.0;
    for (int s = 1; s <= max_splits; ++s) {
      if (active[s] < 1) continue;
      const double waves = std::ceil(static_cast<double>(units) / active[s]);
      const double work = (prefix_tiles + tree_tiles) / static_cast<double>(s) * tile_cost + 3.0;
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

// The kernel's shared-memory limit and its permission for clusters of more than 8
// CTAs, set once on every device that launches it.
template <int D>
cudaError_t set_smem_attr() {
  static PerDeviceOnce attr;
  return attr.run([] {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Layout<D>::kAlloc);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(attn_kernel<D>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return e;
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
  if (set_smem_attr<D>() != cudaSuccess) cudaGetLastError();
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

namespace presto {
namespace pair_attn {

int run_tiles(int B, int N, int Hq, int Hkv, int D, int Tmax) {
  if (B < 1 || N < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv || Tmax < 1 || (D != 64 && D != 128)) return 0;
  const int* active = D == 128 ? active_clusters<128>() : active_clusters<64>();
  const Plan p = make_plan(B, N, Hq, Hkv, Tmax, active);
  const int tiles = (Tmax + kBN - 1) / kBN + (N + kBN - 1) / kBN;
  return (tiles + p.n_splits - 1) / p.n_splits;
}

size_t workspace(int B, int N, int Hq, int Hkv, int D, int Tmax) {
  // KV splits leave partial rows (float32 at most) and fp32 (m, l) for the merge
  const int* active = D == 128 ? active_clusters<128>() : active_clusters<64>();
  const Plan p = make_plan(B, N, Hq, Hkv, Tmax, active);
  if (p.n_splits == 1) return 256;
  return align_up(p.ctas * 2 * kBM * (static_cast<size_t>(D) * 4 + 8), 256);
}

// Arguments as presto_tree_attention's, already checked there.
int launch(const void* q, const void* k_cache, const void* v_cache, const int32_t* kv_len, int Tmax,
           const void* k_tree, const void* v_tree, const uint32_t* mask, const int32_t* n_nodes, int B,
           int N, int Hq, int Hkv, int D, float sm_scale, void* out, float* lse, void* ws,
           size_t ws_bytes, int32_t* dev_status, cudaStream_t stream) {
  const int G = Hq / Hkv;
  const int* active = D == 128 ? active_clusters<128>() : active_clusters<64>();
  const Plan p = make_plan(B, N, Hq, Hkv, Tmax, active);
  Args a{};
  if (p.n_splits > 1) {
    const size_t need = p.ctas * 2 * kBM * (static_cast<size_t>(D) * 4 + 8);
    if (!ws || reinterpret_cast<uintptr_t>(ws) % 16 || ws_bytes < need) return PRESTO_ERR_WORKSPACE;
    a.part_o = static_cast<float2*>(ws);
    a.part_ml = reinterpret_cast<float2*>(static_cast<char*>(ws) + p.ctas * 2 * kBM * D * 4);
  }
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
  a.k_cache = static_cast<const __nv_bfloat16*>(k_cache);
  a.v_cache = static_cast<const __nv_bfloat16*>(v_cache);
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
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.n_splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1] = pdl_attribute();
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  cudaError_t err;
  if (D == 128) {
    if (set_smem_attr<128>() != cudaSuccess) return PRESTO_ERR_CUDA;
    cfg.dynamicSmemBytes = Layout<128>::kAlloc;
    err = cudaLaunchKernelEx(&cfg, attn_kernel<128>, tq, tkc, tvc, tkt, tvt, a);
  } else {
    if (set_smem_attr<64>() != cudaSuccess) return PRESTO_ERR_CUDA;
    cfg.dynamicSmemBytes = Layout<64>::kAlloc;
    err = cudaLaunchKernelEx(&cfg, attn_kernel<64>, tq, tkc, tvc, tkt, tvt, a);
  }
  if (err != cudaSuccess) return PRESTO_ERR_CUDA;
  return launch_status();
}

}  // namespace pair_attn
}  // namespace presto
