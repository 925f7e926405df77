// presto_tree_attention: tree-masked GQA attention of the N tree tokens against the
// committed KV-cache prefix (target verification with a tree-structured attention
// mask, §5.1; App. C (I): each draft token sees the prefix and its ancestors).
//
// The GQA group of one kv head (G = Hq/Hkv query heads x N nodes = G*N rows) is a
// dense contraction against that head's keys, so it runs on the 5th-generation
// tensor cores:
//   * one CTA per (sequence, kv head, 128-row tile, KV split);
//   * warp 8 loads the Q tile, then K tiles of 128 keys into a ring; warp 10 loads V
//     tiles into another (TMA, 128-byte swizzle);
//   * warp 9 issues tcgen05.mma: S_j = Q K_j^T into one of three 128-column TMEM
//     buffers (j mod 3), and O += P_j V_j with P_j (bf16) read from TMEM, where the
//     softmax wrote it over S_j.  QK^T runs up to three KV tiles ahead of PV: the
//     QK^T of tile j + 3 is issued once the PV of tile j (the last reader of that
//     buffer) has completed, so the softmax of the next tiles never waits for the
//     tensor core's commit latency.  The whole warp runs the issue loop and one
//     elected lane issues, so descriptors stay on the uniform datapath;
//   * warps 0-7 run the softmax, two threads per query row (TMEM lane): warps 0-3
//     take score columns 0-63, warps 4-7 columns 64-127 of the same rows.  Each
//     thread masks its 64 scores (prefix length; ancestor bitmask for tree keys; full
//     prefix tiles skip both), the pair combines its row maximum through shared
//     memory (a barrier that also makes a timed-out wait a decision of all eight
//     warps), then exponentiates with packed fp32x2 arithmetic and writes its half
//     of P back over S with tcgen05.st.  The running maximum only moves (and O is
//     rescaled in TMEM, after the previous PV completed) when it grows by more than
//     2^8, so most tiles skip the rescale;
//   * with several KV splits (a row tile's prefix and tree-key tiles dealt out in
//     equal runs; the split count fills the SMs, up to 16), each CTA writes its
//     rows' fp32 (m, l) and O / l to the workspace (bf16 column octets, or float32
//     column pairs when the prefix is short; coalesced either way) and exits.  A
//     second kernel, launched behind it on the stream (programmatic dependent
//     launch: its CTAs start early and wait for the first grid's results), merges
//     the rows over the splits with log-sum-exp weights, 8 rows of a row tile per
//     CTA and all loads of a row issued together.  Splits that are plain CTAs, not
//     a cluster, are not limited by how many clusters of their size fit at once.
// Every wait is bounded; on time-out the CTA records PRESTO_DEV_TIMEOUT, lets its
// copies and MMAs in flight complete (bounded), then frees its TMEM and exits.
#include <cuda_bf16.h>

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

// 11 warps: 0-7 run the softmax (two threads per query row: warps q and q + 4 share
// TMEM lane quadrant q), 8 loads Q and K, 9 issues tensor-core MMAs, 10 loads V
constexpr int kThreads = 352;
constexpr int kKWarp = 8;
constexpr int kMmaWarp = 9;
constexpr int kVWarp = 10;
constexpr int kSoftWarps = 8;
constexpr int kSoftBar = 1;      // named barrier of the softmax warps
constexpr int kSBufs = 3;        // S buffers in TMEM
// TMEM columns: S buffer s (128 fp32) at 128 s, overwritten in place by P (128 bf16
// packed in pairs, its first 64 columns); O (D fp32) at 384
constexpr uint32_t kTmemO = 128 * kSBufs;

struct Args {
  const __nv_bfloat16* k_cache;  // [B, Hkv, Tmax, D] (for the L2 prefetch)
  const __nv_bfloat16* v_cache;
  const int32_t* kv_len;
  const uint32_t* mask;
  const int32_t* n_nodes;
  int B, N, Hq, Hkv, G, Tmax, W, n_mt, n_splits;
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  float2* part_o;   // KV splits: O / l of each row, [CTA][column group][kBM] (groups of
                    // 8 bf16 or, wide partials, 2 float32 columns)
  float2* part_ml;  // KV splits: (m, l) per row [CTA][kBM], log2 domain
  int32_t* dev_status;
};

// Shared memory: the Q tile, the K ring, the V ring.  Every operand is stored as
// 64-column panels of 128-byte rows with the 128-byte swizzle (128 rows per panel).
// Ring depths: K 2 and V 3 at D = 128 (192 KB in all), 4 and 4 at D = 64.
template <int D>
struct Layout {
  static constexpr int kKStages = D == 64 ? 4 : 2;
  static constexpr int kVStages = D == 64 ? 4 : 3;
  static constexpr int kPanels = D / 64;
  static constexpr int kQPanel = kBM * kRowBytes;   // 16 KB
  static constexpr int kKVPanel = kBN * kRowBytes;  // 16 KB
  static constexpr int kQBytes = kBM * D * 2;
  static constexpr int kTileBytes = kBN * D * 2;    // one K or V tile
  static constexpr int kQ = 0;
  static constexpr int kK = kQ + kQBytes;
  static constexpr int kV = kK + kKStages * kTileBytes;
  static constexpr int kBytes = kV + kVStages * kTileBytes;
  static constexpr int kAlloc = kBytes + 1024;  // room to align the base to 1024
};

constexpr int kMaxStages = 4;
struct Bars {
  uint64_t q_full;
  uint64_t k_full[kMaxStages], k_empty[kMaxStages];
  uint64_t v_full[kMaxStages], v_empty[kMaxStages];
  uint64_t s_full[kSBufs], p_full[kSBufs];
  uint64_t o_done;  // one phase per PV: O holds the products of tiles 0..j
  uint64_t drain;   // after a timed-out wait: every MMA issued so far has completed
};

// The softmax warps' barrier with an AND over their predicates: every one of the
// 256 threads arrives, and all leave with the same answer.
__device__ __forceinline__ bool soft_sync_and(bool v) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 q, %1, 0;\n bar.red.and.pred p, %2, %3, q;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(v)), "n"(kSoftBar), "n"(kSoftWarps * 32)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ void soft_sync() {
  asm volatile("bar.sync %0, %1;" ::"n"(kSoftBar), "n"(kSoftWarps * 32) : "memory");
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
  __shared__ float xmax[2][2][kBM];  // per iteration parity and half: the half-row maxima
  __shared__ float xl[2][kBM];       // per half: the half-row sums

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int idx = blockIdx.x;
  const int split = idx % a.n_splits;
  idx /= a.n_splits;
  const int mt = idx % a.n_mt;  // row tile
  idx /= a.n_mt;
  const int g = idx % a.Hkv;
  const int b = idx / a.Hkv;
  const bool partial = a.n_splits > 1;  // KV splits: this CTA leaves a partial result
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
    for (int s = 0; s < kSBufs; ++s) {
      mbar_init(&bars.s_full[s], 1);
      mbar_init(&bars.p_full[s], kSoftWarps);
    }
    mbar_init(&bars.o_done, 1);
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
  // No kernel of the round writes the KV cache or kv_len (the caller does, between
  // rounds), so the split's KV tiles and their KV-cache part are known before the
  // dependency wait: the loaders fill their rings with KV-cache tiles and the rest of
  // the split's range is asked of L2 while the previous kernels still run.  q and the
  // tree K/V (computed from the tree, in a real round, by the target model), the
  // ancestor mask and the node count are read only after griddepcontrol.wait.
  const int kv_raw = ld_chain(a.kv_len + b);
  int kv = kv_raw;
  if (kv < 0 || kv > a.Tmax) {
    if (tid == 0) report(a.dev_status, PRESTO_DEV_BAD_KVLEN);
    kv = kv < 0 ? 0 : a.Tmax;
  }
  // split partials in float32 when the prefix is short: then a row averages few keys,
  // its values can be as large as single V entries, and the bf16 roundings of P, of a
  // bf16 partial and of the output could together reach 2e-2 of N(0, 1) values; with
  // a long prefix bf16 partials (half the merge traffic) lose nothing measurable
  const bool wide = kv < kWidePartialKeys;
  const int prefix_tiles = (kv + kBN - 1) / kBN;
  // the KV tiles of a row tile, prefix tiles then tree tiles, in equal runs over the
  // splits: this split's local tile j is prefix tile t_begin + j for j < n_prefix,
  // else tree tile tree0 + (j - n_prefix).  The tree tiles cover the node budget N
  // (the built node count is not known before the wait); keys past it are masked out.
  const int tree_tiles = (a.N + kBN - 1) / kBN;
  const int total = prefix_tiles + tree_tiles;
  const int per = (total + a.n_splits - 1) / a.n_splits;
  const int t_begin = min(split * per, total);
  const int nt = min(total, t_begin + per) - t_begin;  // KV tiles of this split (CTA-uniform)
  const int n_prefix = max(0, min(nt, prefix_tiles - t_begin));
  const int tree0 = t_begin + n_prefix - prefix_tiles;
  constexpr int kRing = Ly::kKStages < Ly::kVStages ? Ly::kKStages : Ly::kVStages;
  if (tid == 0 && n_prefix > kRing) {  // the prefix tiles beyond the rings, into L2
    const size_t row0 = (static_cast<size_t>(b) * a.Hkv + g) * a.Tmax;
    const int t0 = (t_begin + kRing) * kBN, t1 = min((t_begin + n_prefix) * kBN, kv);
    if (t1 > t0) {
      const uint32_t bytes = static_cast<uint32_t>(t1 - t0) * D * 2u;
      prefetch_l2_bulk(a.k_cache + (row0 + t0) * D, bytes);
      prefetch_l2_bulk(a.v_cache + (row0 + t0) * D, bytes);
    }
  }

  volatile int* abort = &abort_flag;
  auto fail = [&]() {
    *abort = 1;
    report(a.dev_status, PRESTO_DEV_TIMEOUT);
  };

  int issued = 0;         // K or V tiles this warp's lane 0 has issued (the loaders)
  bool q_issued = false;  // the K loader has issued the Q tile
  if (nt > 0 && warp == kKWarp) {
    // ------------------------------------------------------------ Q and K loads
    if (lane == 0) {
      prefetch_tensormap(&tm_q);
      prefetch_tensormap(&tm_kc);
      prefetch_tensormap(&tm_kt);
      // K_j -> slot j % Ly::kKStages, once the QK^T of K_{j - Ly::kKStages} completed;
      // the first KV-cache tiles before the dependency wait, Q and the rest after it
      const int early = min(n_prefix, Ly::kKStages);
      for (int j = 0; j < nt; ++j) {
        if (j == early) {
          pdl_wait();
          mbar_arrive_expect_tx(&bars.q_full, Ly::kQBytes);
          for (int p = 0; p < Ly::kPanels; ++p)
            tma_load_3d(smem + Ly::kQ + p * Ly::kQPanel, &tm_q, p * 64, g * a.G,
                        b * a.N + mt * nodes_per_tile, &bars.q_full);
          q_issued = true;
        }
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
      if (!q_issued) {  // every tile was an early one
        pdl_wait();
        mbar_arrive_expect_tx(&bars.q_full, Ly::kQBytes);
        for (int p = 0; p < Ly::kPanels; ++p)
          tma_load_3d(smem + Ly::kQ + p * Ly::kQPanel, &tm_q, p * 64, g * a.G,
                      b * a.N + mt * nodes_per_tile, &bars.q_full);
        q_issued = true;
      }
    }
  } else if (nt > 0 && warp == kVWarp) {
    // ------------------------------------------------------------ V loads
    if (lane == 0) {
      prefetch_tensormap(&tm_vc);
      prefetch_tensormap(&tm_vt);
      // V_j -> slot j % Ly::kVStages, once the PV of V_{j - Ly::kVStages} completed;
      // the first KV-cache tiles before the dependency wait
      const int early = min(n_prefix, Ly::kVStages);
      for (int j = 0; j < nt; ++j) {
        if (j == early) pdl_wait();
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
    // S_j goes to TMEM buffer j % 3.  The first three QK^T are issued as their K tiles
    // land; then per tile j: PV_j once P_j is written (P_j read from buffer j % 3),
    // and QK^T of tile j + 3 into the same buffer once PV_j has completed (o_done),
    // so S is never rewritten while P is still being read.  The whole warp runs this
    // loop (wait outcomes made warp-uniform); one elected lane issues each MMA and
    // commit.
    constexpr uint32_t idesc_qk = idesc_bf16_f32(kBM, kBN, false);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, D, true);
    const uint64_t q_desc = smem_desc_sw128(smem_u32(smem + Ly::kQ), 16, 1024);
    const uint64_t k_desc0 = smem_desc_sw128(smem_u32(smem + Ly::kK), 16, 1024);
    const uint64_t v_desc0 = smem_desc_sw128(smem_u32(smem + Ly::kV), Ly::kKVPanel, 1024);
    auto wait = [&](uint64_t* bar, uint32_t parity) {
      const bool ok = __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
      if (ok) tc_fence_after();
      return ok;
    };
    // S_j = Q K_j^T (K_j resident)
    auto qk = [&](int j) {
      const int s = j % kSBufs;
      // descriptor start addresses are in 16-byte units in the low bits
      const uint64_t kd = k_desc0 + (((j % Ly::kKStages) * Ly::kTileBytes) >> 4);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t qo = ((kk >> 2) * Ly::kQPanel + (kk & 3) * 32) >> 4;
        const uint32_t ko = ((kk >> 2) * Ly::kKVPanel + (kk & 3) * 32) >> 4;
        mma_bf16_warp(tmem_base + s * 128, q_desc + qo, kd + ko, idesc_qk, kk > 0);
      }
      mma_commit_warp(&bars.s_full[s]);
      mma_commit_warp(&bars.k_empty[j % Ly::kKStages]);
    };
    // O (+)= P_j V_j, P_j read from TMEM (8 columns = 16 keys per step)
    auto pv = [&](int j) {
      const int s = j % kSBufs;
      if (!wait(&bars.p_full[s], (j / kSBufs) & 1)) return false;
      const uint64_t vd = v_desc0 + (((j % Ly::kVStages) * Ly::kTileBytes) >> 4);
#pragma unroll
      for (int kk = 0; kk < kBN / 16; ++kk)
        mma_bf16_ts_warp(tmem_base + kTmemO, tmem_base + s * 128 + kk * 8,
                         vd + ((kk * 16 * kRowBytes) >> 4), idesc_pv, (j > 0 || kk > 0) ? 1u : 0u);
      mma_commit_warp(&bars.o_done);
      mma_commit_warp(&bars.v_empty[j % Ly::kVStages]);
      return true;
    };
    bool ok = wait(&bars.q_full, 0);
    for (int j = 0; ok && j < min(nt, kSBufs); ++j) {
      ok = wait(&bars.k_full[j % Ly::kKStages], (j / Ly::kKStages) & 1);
      if (ok) qk(j);
    }
    for (int j = 0; ok && j < nt; ++j) {
      ok = wait(&bars.v_full[j % Ly::kVStages], (j / Ly::kVStages) & 1) && pv(j);
      const int jn = j + kSBufs;
      if (ok && jn < nt) {
        ok = wait(&bars.o_done, j & 1) &&
             wait(&bars.k_full[jn % Ly::kKStages], (jn / Ly::kKStages) & 1);
        if (ok) qk(jn);
      }
    }
    if (!ok && lane == 0) fail();
  } else if (nt > 0 && warp < kSoftWarps) {
    // ------------------------------------------------------------ softmax warps
    const int quad = warp & 3;        // TMEM lane quadrant
    const int h = warp >> 2;          // half of the score columns: 64 h .. 64 h + 63
    const int r = quad * 32 + lane;   // row of the tile
    const uint32_t lane_addr = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t tO = tmem_base + kTmemO + lane_addr;
    const int node = mt * nodes_per_tile + r / a.G;
    const uint32_t* mrow =
        node < a.N ? a.mask + (static_cast<size_t>(b) * a.N + node) * a.W : nullptr;
    pdl_wait();  // the mask and the node count come from the build
    const int nn = min(max(ld_chain(a.n_nodes + b), 0), a.N);
    float m = -INFINITY, l = 0.f;  // m: running (possibly stale) max, log2 domain; l: this half's sum
    bool ok = true;
    for (int j = 0; j < nt; ++j) {
      const int s = j % kSBufs;
      const uint32_t tS = tmem_base + s * 128 + lane_addr;  // S_j, then P_j in place
      // wait outcomes are warp-uniform (tcgen05.ld needs the whole warp) and then
      // shared by all eight warps at the exchange barrier below
      bool got = ok && __all_sync(0xffffffffu, mbar_wait(&bars.s_full[s], (j / kSBufs) & 1, abort));
      if (ok && !got) fail();  // the other warps' waits end at once
      float v[64];
      float mx = -INFINITY;
      const bool full = j < n_prefix && kv - (t_begin + j) * kBN >= kBN;  // CTA-uniform
      if (got) {
        tc_fence_after();
        // masks of this half's two 32-key chunks: prefix keys beyond kv_len; tree keys
        // outside the ancestor set (a full prefix tile needs none)
        uint32_t bits[2];
        if (j < n_prefix) {
          const int lim = kv - (t_begin + j) * kBN - 64 * h;
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            const int lc = lim - 32 * c;
            bits[c] = lc >= 32 ? 0xffffffffu : (lc <= 0 ? 0u : (1u << lc) - 1u);
          }
        } else {
          const int wi = (((tree0 + j - n_prefix) * kBN) >> 5) + 2 * h;
#pragma unroll
          for (int c = 0; c < 2; ++c) bits[c] = (mrow && wi + c < a.W) ? ld_chain(mrow + wi + c) : 0u;
        }
        // this half's 64 scores: two loads in flight, one wait
#pragma unroll
        for (int c = 0; c < 2; ++c)
          tmem_ld32(tS + 64 * h + c * 32, *reinterpret_cast<float(*)[32]>(v + 32 * c));
        tmem_wait_ld();
        if (!full) {  // masked scores -> -inf (exp2 of -inf is 0)
#pragma unroll
          for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int e = 0; e < 32; ++e) v[32 * c + e] = ((bits[c] >> e) & 1u) ? v[32 * c + e] : -INFINITY;
        }
        mx = fmaxf(row_max32(v), row_max32(v + 32)) * a.scale_log2;  // scale > 0 commutes with max
        xmax[j & 1][h][r] = mx;
      }
      // both halves' maxima are written and every load of S_j has completed (the
      // other half overwrites part of this half's S columns with its P below)
      tc_fence_before();
      got = soft_sync_and(got);
      tc_fence_after();
      if (!got) {
        ok = false;
        break;
      }
      mx = fmaxf(mx, xmax[j & 1][h ^ 1][r]);
      // stale-max online softmax: move m only when the row max exceeds it by > 2^8
      // (both halves of a row take the same decision)
      const bool move = mx > m + kRescaleLog2;
      const float alpha = move ? ex2(m - mx) : 1.f;
      if (move) m = mx;
      const float m_use = m == -INFINITY ? 0.f : m;
      // p = exp2(s * scale - m), stored as bf16 pairs over the S columns: this half's
      // 64 keys are P columns 32 h .. 32 h + 31; the half-row sum in packed chains
      const uint64_t sc2 = pack2(a.scale_log2, a.scale_log2), nm2 = pack2(-m_use, -m_use);
      uint64_t acc[2] = {0ull, 0ull};
#pragma unroll
      for (int c = 0; c < 2; ++c) {
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
        tmem_st16(tS + 32 * h + c * 16, pk);
      }
      if (j > 0 && __any_sync(0xffffffffu, move)) {
        // O *= alpha over this half's columns (rows that did not move: 1), once the
        // PV of tile j - 1 has completed
        if (__all_sync(0xffffffffu, mbar_wait(&bars.o_done, (j - 1) & 1, abort))) {
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < D / 64; ++c) {
            float o[32];
            const uint32_t col = (D / 2) * h + c * 32;
            tmem_ld32(tO + col, o);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] *= alpha;
            tmem_st32(tO + col, o);
          }
        } else {
          ok = false;  // the next exchange barrier makes it every warp's decision
          fail();
        }
      }
      float rs, rs1;
      unpack2(add2(acc[0], acc[1]), rs, rs1);
      l = l * alpha + (rs + rs1);
      tmem_wait_st();  // P (and a rescaled O) are in TMEM before the MMA is released
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars.p_full[s]);
    }
    // the row's sum over both halves
    xl[h][r] = l;
    soft_sync();
    l += xl[h ^ 1][r];
    if (ok) {
      ok = __all_sync(0xffffffffu, mbar_wait(&bars.o_done, (nt - 1) & 1, abort));
      if (!ok) fail();
    }
    if (partial) {
      // this split's normalised row and (m, l) for the merge (a failed or empty row
      // is marked by m = -inf and contributes nothing); each half writes its columns
      const size_t prow = static_cast<size_t>(blockIdx.x) * kBM + r;
      if (h == 0) a.part_ml[prow] = ok ? make_float2(m, l) : make_float2(-INFINITY, 0.f);
      if (ok) {
        tc_fence_after();
        // the row normalised by its own l (values stay within the range of V), laid
        // out so that a warp's 32 rows of one column group are contiguous: bf16
        // column octets (512 bytes), or float32 column pairs (256 bytes) when the
        // sequence's prefix is short (wide partials)
        const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll 1
        for (int cc = 0; cc < D / 64; ++cc) {
          const int c = h * (D / 64) + cc;  // 32-column chunk of O
          float o[32];
          tmem_ld32(tO + c * 32, o);
          tmem_wait_ld();
          if (wide) {
            float2* dst = reinterpret_cast<float2*>(a.part_o) +
                          static_cast<size_t>(blockIdx.x) * (D / 2) * kBM + r;
#pragma unroll
            for (int q = 0; q < 16; ++q)
              dst[(c * 16 + q) * kBM] = make_float2(o[q * 2] * inv, o[q * 2 + 1] * inv);
          } else {
            uint4* dst = reinterpret_cast<uint4*>(a.part_o) +
                         static_cast<size_t>(blockIdx.x) * (D / 8) * kBM + r;
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
              dst[(c * 4 + q) * kBM] = w4;
            }
          }
        }
      }
    } else if (ok) {
      tc_fence_after();
      // the normalised bf16 row (this half's columns), and its lse
      const int hh = r % a.G;
      const bool used = node < a.N && node < nn && l > 0.f;
      const float inv = used ? 1.f / l : 0.f;
      __nv_bfloat16* orow =
          a.out + ((static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh) * D;
#pragma unroll 1
      for (int cc = 0; cc < D / 64; ++cc) {
        const int c = h * (D / 64) + cc;
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
      if (h == 0 && node < a.N && a.lse)
        a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh] =
            used ? (m + log2f(l)) * kLn2 : -INFINITY;
    }
  }

  // every thread past the dependency wait before the outputs and the merge (which read
  // the node count); a thread that already waited returns at once
  pdl_wait();

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
      if (warp == kKWarp && q_issued) mbar_wait(&bars.q_full, 0, nullptr);
      for (int j = max(0, issued - S); j < issued; ++j) mbar_wait(&full[j % S], (j / S) & 1, nullptr);
    }
    if (nt > 0 && warp == kMmaWarp) {
      mma_commit_warp(&bars.drain);
      mbar_wait(&bars.drain, 0, nullptr);
    }
  }

  if (partial) {
    if (nt == 0 && tid < kBM)  // an empty split contributes nothing
      a.part_ml[static_cast<size_t>(blockIdx.x) * kBM + tid] = make_float2(-INFINITY, 0.f);
  } else if (nt == 0 && tid < kBM) {  // no keys at all: a zero row, lse -inf
    const int r = tid;
    const int node = mt * nodes_per_tile + r / a.G, hh = r % a.G;
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
}

// ---------------------------------------------------------------- split merge
// One CTA per kMergeRows rows of a row tile: the KV splits of the row tile (CTAs
// cta0 .. cta0 + n_splits - 1 of attn_kernel) have left each row's (m, l) and
// normalised O in the workspace, and the rows are combined with log-sum-exp weights
// (the partials stay in L2).  Launched right behind attn_kernel with programmatic
// dependent launch: the CTAs may start while it runs and wait for its results.
constexpr int kMergeRows = 8;
constexpr int kMergeThreads = 256;
static_assert(kBM % kMergeRows == 0, "a row tile is whole merge slices");

template <int D>
__global__ void __launch_bounds__(kMergeThreads) attn_merge_kernel(const Args a) {
  __shared__ float mw[kMergeRows][kMaxSplits + 1];  // per-row weights over the splits
  __shared__ float mlse[kMergeRows];                // per-row lse
  constexpr int kThreads = kMergeThreads;  // the merge body's block size
  constexpr int kSlices = kBM / kMergeRows;
  const int tid = threadIdx.x;
  int idx = blockIdx.x;
  const int slice = idx % kSlices;
  idx /= kSlices;
  const int mt = idx % a.n_mt;
  idx /= a.n_mt;
  const int g = idx % a.Hkv;
  const int b = idx / a.Hkv;
  const int nodes_per_tile = kBM / a.G;
  pdl_launch_dependents();
  // the partials' precision, as attn_kernel chose it (which reports a bad kv_len);
  // no kernel of a round writes kv_len, so it is read before the dependency wait and
  // the partial loads after it are the merge's only round trip
  int kv = ld_chain(a.kv_len + b);
  kv = kv < 0 ? 0 : (kv > a.Tmax ? a.Tmax : kv);
  const bool wide = kv < kWidePartialKeys;
  pdl_wait();  // the partials come from attn_kernel (and the node count from the build)
  const int nn = min(max(ld_chain(a.n_nodes + b), 0), a.N);
  const int nsp = a.n_splits;
  const size_t cta0 = ((static_cast<size_t>(b) * a.Hkv + g) * a.n_mt + mt) * nsp;
  const int r0 = slice * kMergeRows;
  const int nr = kMergeRows;
  // One item = one row of the slice x one column group (a bf16 octet or a float32
  // pair), rows fastest (coalesced partial loads).  Each thread's first items are
  // loaded before the per-row weights are formed (one thread per row, into shared
  // memory), so the usual case costs one L2 round trip.
  auto merge = [&](auto wide_tag) {
    constexpr bool kWide = decltype(wide_tag)::value;
    using PT = std::conditional_t<kWide, float2, uint4>;
    constexpr int kCG = kWide ? D / 2 : D / 8;  // column groups per row
    const PT* part = reinterpret_cast<const PT*>(a.part_o);
    const int nitems = nr * kCG;
    auto load_item = [&](int item, PT (&o)[kMaxSplits]) {
      const int cg = item / max(nr, 1), row = r0 + item % max(nr, 1);
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s)
        o[s] = (item < nitems && s < nsp) ? __ldcg(part + ((cta0 + s) * kCG + cg) * kBM + row)
                                         : PT{};
    };
    // items loaded before the weights: two of the float32 pairs, one of the bf16
    // octets (a slice has at most one octet item per thread at D = 128)
    constexpr int kAhead = kWide ? 2 : 1;
    PT oa[kMaxSplits], ob[kMaxSplits];
    load_item(tid, oa);
    if constexpr (kAhead > 1) load_item(tid + kThreads, ob);
    if (tid < nr) {
      // the row's weights over the splits, w_s l_s / L (a split without keys for the
      // row has m = -inf and weight 0), and its lse
      const int row = r0 + tid;
      float2 ml[kMaxSplits];
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s)
        ml[s] = s < nsp ? __ldcg(a.part_ml + (cta0 + s) * kBM + row) : make_float2(-INFINITY, 0.f);
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
      const int node = mt * nodes_per_tile + row / a.G;
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
      const int node = mt * nodes_per_tile + row / a.G;
      const int hh = row % a.G;
      if (node >= a.N) return;
      float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
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
            const uint32_t ow[4] = {o[s].x, o[s].y, o[s].z, o[s].w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              acc[2 * e] = fmaf(w, __uint_as_float(ow[e] << 16), acc[2 * e]);
              acc[2 * e + 1] = fmaf(w, __uint_as_float(ow[e] & 0xffff0000u), acc[2 * e + 1]);
            }
          }
        }
      }
      const size_t orow = ((static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh) * D;
      if constexpr (kWide) {
        *reinterpret_cast<__nv_bfloat162*>(a.out + orow + cg * 2) = __floats2bfloat162_rn(acc[0], acc[1]);
      } else {
        uint4 w4;
        uint32_t* w = reinterpret_cast<uint32_t*>(&w4);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const __nv_bfloat162 o2 = __floats2bfloat162_rn(acc[2 * e], acc[2 * e + 1]);
          w[e] = *reinterpret_cast<const uint32_t*>(&o2);
        }
        *reinterpret_cast<uint4*>(a.out + orow + cg * 8) = w4;
      }
      if (cg == 0 && a.lse) a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + g * a.G + hh] = mlse[i];
    };
    finish_item(tid, oa);
    if constexpr (kAhead > 1) finish_item(tid + kThreads, ob);
    for (int item = tid + kAhead * kThreads; item < nitems; item += kThreads) {
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
  int G, n_mt, n_splits;
  size_t ctas;
};

// resident = how many CTAs of the kernel the GPU holds at once.
Plan make_plan(int B, int N, int Hq, int Hkv, int Tmax, int resident) {
  Plan p;
  p.G = Hq / Hkv;
  p.n_mt = (N * p.G + kBM - 1) / kBM;
  const int tiles = (Tmax + kBN - 1) / kBN + (N + kBN - 1) / kBN;
  int max_splits = tiles / 2 > 1 ? tiles / 2 : 1;
  if (max_splits > kMaxSplits) max_splits = kMaxSplits;
  // The split count by the estimated time: waves of resident row tiles (each s
  // CTAs) x (KV tiles of the busiest CTA -- the tiles are dealt out in runs of
  // ceil(tiles / s) -- plus a fixed cost of about three tiles), lightly penalising
  // splits (each adds rows to merge), so that of two split counts with the same runs
  // the smaller wins.
  const long long units = static_cast<long long>(B) * Hkv * p.n_mt;
  double best_cost = 1e30;
  p.n_splits = 1;
  for (int s = 1; s <= max_splits; ++s) {
    const int active = resident / s;
    if (active < 1) continue;
    const double waves = std::ceil(static_cast<double>(units) / active);
    const int run = (tiles + s - 1) / s;
    const double cost = waves * (run + 3.0) * (1.0 + 0.02 * (s - 1));
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      p.n_splits = s;
    }
  }
  p.ctas = static_cast<size_t>(units) * p.n_splits;
  return p;
}

// The kernel's shared-memory limit, set once on every device that launches it.
template <int D>
cudaError_t set_smem_attr() {
  static PerDeviceOnce attr;
  return attr.run([] {
    return cudaFuncSetAttribute(attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                Layout<D>::kAlloc);
  });
}

// CTAs of the kernel resident on the GPU at once (queried once per device and D;
// one SM's worth if the query fails).
template <int D>
int resident_ctas() {
  static int cached[kMaxDevices];
  static bool done[kMaxDevices] = {false};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) dev = 0;
  std::lock_guard<std::mutex> lock(mu);
  if (done[dev]) return cached[dev];
  int per_sm = 0;
  if (set_smem_attr<D>() != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, attn_kernel<D>, kThreads,
                                                    Layout<D>::kAlloc) != cudaSuccess) {
    cudaGetLastError();
    per_sm = 0;
  }
  cached[dev] = per_sm > 0 ? per_sm * sm_count() : 1;
  done[dev] = true;
  return cached[dev];
}

}  // namespace

// The long-run schedule (tree_attention_pair.cu): two row tiles per CTA in ping-pong.
// Over a long run of KV tiles per CTA the two tiles' softmax-to-tensor-core chains
// interleave and beat this file's deeper S pipeline for one tile; over a short run
// (the small rounds) this file's schedule wins, mostly in the fill and the merge.
namespace pair_attn {
int run_tiles(int B, int N, int Hq, int Hkv, int D, int Tmax);  // KV tiles per CTA of its plan
size_t workspace(int B, int N, int Hq, int Hkv, int D, int Tmax);
int launch(const void* q, const void* k_cache, const void* v_cache, const int32_t* kv_len, int Tmax,
           const void* k_tree, const void* v_tree, const uint32_t* mask, const int32_t* n_nodes, int B,
           int N, int Hq, int Hkv, int D, float sm_scale, void* out, float* lse, void* ws,
           size_t ws_bytes, int32_t* dev_status, cudaStream_t stream);
}  // namespace pair_attn

constexpr int kPairMinRun = 8;  // KV tiles per CTA from which the pair schedule is taken

bool use_pair(int B, int N, int Hq, int Hkv, int D, int Tmax) {
  return pair_attn::run_tiles(B, N, Hq, Hkv, D, Tmax) >= kPairMinRun;
}

}  // namespace presto

using namespace presto;

extern "C" size_t presto_attn_workspace(int B, int N, int Hq, int Hkv, int D, int Tmax) {
  if (B < 1 || N < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv || Tmax < 1 || (D != 64 && D != 128))
    return 0;
  if (use_pair(B, N, Hq, Hkv, D, Tmax)) return pair_attn::workspace(B, N, Hq, Hkv, D, Tmax);
  // KV splits leave partial rows (float32 at most) and fp32 (m, l) for the merge
  const int resident = D == 128 ? resident_ctas<128>() : resident_ctas<64>();
  const Plan p = make_plan(B, N, Hq, Hkv, Tmax, resident);
  if (p.n_splits == 1) return 256;
  return align_up(p.ctas * kBM * (static_cast<size_t>(D) * 4 + 8), 256);
}

extern "C" int presto_attn_launches(int B, int N, int Hq, int Hkv, int D, int Tmax) {
  if (B < 1 || N < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv || Tmax < 1 || (D != 64 && D != 128))
    return 0;
  if (use_pair(B, N, Hq, Hkv, D, Tmax)) return 1;
  const int resident = D == 128 ? resident_ctas<128>() : resident_ctas<64>();
  return make_plan(B, N, Hq, Hkv, Tmax, resident).n_splits > 1 ? 2 : 1;
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
  if (use_pair(B, N, Hq, Hkv, D, Tmax))
    return pair_attn::launch(q, k_cache, v_cache, kv_len, Tmax, k_tree, v_tree, mask, n_nodes, B, N,
                             Hq, Hkv, D, sm_scale, out, lse, ws, ws_bytes, dev_status, stream);
  const int resident = D == 128 ? resident_ctas<128>() : resident_ctas<64>();
  const Plan p = make_plan(B, N, Hq, Hkv, Tmax, resident);
  Args a{};
  if (p.n_splits > 1) {
    const size_t need = p.ctas * kBM * (static_cast<size_t>(D) * 4 + 8);
    if (!ws || reinterpret_cast<uintptr_t>(ws) % 16 || ws_bytes < need) return PRESTO_ERR_WORKSPACE;
    a.part_o = static_cast<float2*>(ws);
    a.part_ml = reinterpret_cast<float2*>(static_cast<char*>(ws) + p.ctas * kBM * D * 4);
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
  attr[0] = pdl_attribute();
  cfg.attrs = attr;
  cfg.numAttrs = 1;
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
  if (p.n_splits > 1) {  // the merge of the splits, right behind on the stream
    cudaLaunchConfig_t mc{};
    mc.gridDim = dim3(static_cast<unsigned>(p.ctas / p.n_splits) * (kBM / kMergeRows));
    mc.blockDim = dim3(kMergeThreads);
    mc.stream = stream;
    mc.attrs = attr;
    mc.numAttrs = 1;
    err = D == 128 ? cudaLaunchKernelEx(&mc, attn_merge_kernel<128>, a)
                   : cudaLaunchKernelEx(&mc, attn_merge_kernel<64>, a);
    if (err != cudaSuccess) return PRESTO_ERR_CUDA;
  }
  return launch_status();
}

