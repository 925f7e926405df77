// presto_tree_attention: tree-masked GQA attention of the N tree tokens against the
// committed KV-cache prefix (target verification with a tree-structured attention
// mask, §5.1; App. C (I): each draft token sees the prefix and its ancestors).
//
// The GQA group of one kv head (G = Hq/Hkv query heads x N nodes = G*N rows) is a
// dense contraction against that head's keys, so it runs on the 5th-generation
// tensor cores:
//   * one CTA per (sequence, kv head, 128-row M tile, KV split);
//   * warp 0 issues TMA loads (Q once, then K/V tiles of 128 keys, double buffered);
//   * warp 1 issues tcgen05.mma: S = Q K^T into TMEM (128 fp32 columns), and after
//     softmax O += P V into TMEM (D fp32 columns);
//   * warps 2-5 (one thread per TMEM lane = query row) read S with tcgen05.ld,
//     apply the prefix-length and ancestor-bitmask masks, run the online softmax,
//     write P (bf16, 128-byte swizzled K-major) to shared memory and rescale O in
//     TMEM when the row maximum grows;
//   * with several KV splits per row block, each CTA writes (O, m, l) partials and
//     a combine kernel merges them (log-sum-exp weighting).
// Every wait is bounded; on time-out the CTA records PRESTO_DEV_TIMEOUT and unwinds.
#include <cuda_bf16.h>

#include <cudaTypedefs.h>

#include <cmath>
#include <initializer_list>
#include <mutex>

#include "common.cuh"

namespace presto {
namespace {

constexpr int kBM = 128;        // query rows per tile (TMEM lanes)
constexpr int kBN = 128;        // keys per tile
constexpr int kThreads = 192;   // 6 warps
constexpr int kPanelBytes = 128 * 128;  // 128 rows x 128 bytes (64 bf16)
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr uint32_t kTmemCols = 256;

struct Args {
  const int32_t* kv_len;
  const uint32_t* mask;
  const int32_t* n_nodes;
  int B, N, Hq, Hkv, G, Tmax, W, n_mt, n_splits;
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  float* ws_o;     // [cta][128][D] unnormalised O (splits > 1)
  float2* ws_ml;   // [cta][128] (m, l), log2 domain
  int32_t* dev_status;
};

template <int D>
struct Layout {
  static constexpr int kPanels = D / 64;
  static constexpr int kQBytes = kBM * D * 2;
  static constexpr int kTileBytes = kBN * D * 2;
  static constexpr int kPBytes = kBM * kBN * 2;
  static constexpr int kQ = 0;
  static constexpr int kK0 = kQ + kQBytes;
  static constexpr int kV0 = kK0 + 2 * kTileBytes;
  static constexpr int kP = kV0 + 2 * kTileBytes;
  static constexpr int kBytes = kP + kPBytes;
  static constexpr int kAlloc = kBytes + 1024;  // room to align the base to 1024
};

struct Bars {
  uint64_t q_full;
  uint64_t kv_full[2];
  uint64_t kv_empty[2];
  uint64_t s_full;
  uint64_t s_free;
  uint64_t p_full;
  uint64_t o_done;
};

// Per-row epilogue shared by the direct path and the partial path.
template <int D>
__device__ __forceinline__ void write_row(const Args& a, int b, int g, int node, int hh, int nn,
                                          const float* o, float m, float l) {
  if (node >= a.N) return;
  const int h = g * a.G + hh;
  __nv_bfloat16* dst = a.out + ((static_cast<size_t>(b) * a.N + node) * a.Hq + h) * D;
  const bool used = node < nn && l > 0.f;
  const float inv = used ? 1.f / l : 0.f;
#pragma unroll
  for (int c = 0; c < D; c += 8) {
    uint4 u;
    uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const __nv_bfloat162 v =
          __floats2bfloat162_rn(used ? o[c + 2 * e] * inv : 0.f, used ? o[c + 2 * e + 1] * inv : 0.f);
      w[e] = *reinterpret_cast<const uint32_t*>(&v);
    }
    *reinterpret_cast<uint4*>(dst + c) = u;
  }
  if (a.lse)
    a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + h] =
        used ? (m + log2f(l)) * kLn2 : -INFINITY;
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
  const int mt = idx % a.n_mt;
  idx /= a.n_mt;
  const int g = idx % a.Hkv;
  const int b = idx / a.Hkv;

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
  const int rows_per_node = a.G;
  const int node0 = mt * (kBM / rows_per_node);

  if (nt == 0) {  // nothing to attend to in this split (CTA-uniform)
    if (tid < kBM) {
      const int node = node0 + tid / a.G, hh = tid % a.G;
      if (a.n_splits > 1) {
        a.ws_ml[static_cast<size_t>(blockIdx.x) * kBM + tid] = make_float2(-INFINITY, 0.f);
      } else {
        float zero[D];
#pragma unroll
        for (int c = 0; c < D; ++c) zero[c] = 0.f;
        write_row<D>(a, b, g, node, hh, nn, zero, -INFINITY, 0.f);
      }
    }
    return;
  }

  uint8_t* sQ = smem + Ly::kQ;
  uint8_t* sP = smem + Ly::kP;

  if (tid == 0) {
    mbar_init(&bars.q_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars.kv_full[s], 1);
      mbar_init(&bars.kv_empty[s], 1);
    }
    mbar_init(&bars.s_full, 1);
    mbar_init(&bars.s_free, kBM);
    mbar_init(&bars.p_full, kBM);
    mbar_init(&bars.o_done, 1);
    abort_flag = 0;
    fence_barrier_init();
    prefetch_tensormap(&tm_q);
    prefetch_tensormap(&tm_kc);
    prefetch_tensormap(&tm_vc);
    prefetch_tensormap(&tm_kt);
    prefetch_tensormap(&tm_vt);
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tS = tmem_base;
  const uint32_t tO = tmem_base + 128;
  volatile int* abort = &abort_flag;
  auto fail = [&]() {
    *abort = 1;
    report(a.dev_status, PRESTO_DEV_TIMEOUT);
  };

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      mbar_arrive_expect_tx(&bars.q_full, Ly::kQBytes);
      for (int p = 0; p < Ly::kPanels; ++p)
        tma_load_3d(sQ + p * kPanelBytes, &tm_q, p * 64, g * a.G, b * a.N + node0, &bars.q_full);
      for (int j = 0; j < nt; ++j) {
        const int st = j & 1;
        if (j >= 2 && !mbar_wait(&bars.kv_empty[st], ((j - 2) >> 1) & 1, abort)) {
          fail();
          break;
        }
        uint8_t* sK = smem + Ly::kK0 + st * Ly::kTileBytes;
        uint8_t* sV = smem + Ly::kV0 + st * Ly::kTileBytes;
        mbar_arrive_expect_tx(&bars.kv_full[st], 2 * Ly::kTileBytes);
        if (j < n_prefix) {
          const int t0 = (t_begin + j) * kBN;
          for (int p = 0; p < Ly::kPanels; ++p) {
            tma_load_3d(sK + p * kPanelBytes, &tm_kc, p * 64, t0, b * a.Hkv + g, &bars.kv_full[st]);
            tma_load_3d(sV + p * kPanelBytes, &tm_vc, p * 64, t0, b * a.Hkv + g, &bars.kv_full[st]);
          }
        } else {
          const int j0 = (j - n_prefix) * kBN;
          for (int p = 0; p < Ly::kPanels; ++p) {
            tma_load_3d(sK + p * kPanelBytes, &tm_kt, p * 64, g, b * a.N + j0, &bars.kv_full[st]);
            tma_load_3d(sV + p * kPanelBytes, &tm_vt, p * 64, g, b * a.N + j0, &bars.kv_full[st]);
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(kBM, kBN, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, D, true);
      const uint32_t q_addr = smem_u32(sQ);
      const uint32_t p_addr = smem_u32(sP);
      auto issue_qk = [&](int j) {
        const uint32_t k_addr = smem_u32(smem + Ly::kK0 + (j & 1) * Ly::kTileBytes);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          mma_bf16(tS, smem_desc_sw128(q_addr + off, 16, 1024),
                   smem_desc_sw128(k_addr + off, 16, 1024), idesc_qk, kk > 0);
        }
        mma_commit(&bars.s_full);
      };
      bool ok = mbar_wait(&bars.q_full, 0, abort) && mbar_wait(&bars.kv_full[0], 0, abort);
      if (ok) {
        tc_fence_after();
        issue_qk(0);
      }
      for (int j = 0; ok && j < nt; ++j) {
        if (j + 1 < nt) {
          // S may be overwritten once every softmax thread has read S_j.
          ok = mbar_wait(&bars.kv_full[(j + 1) & 1], ((j + 1) >> 1) & 1, abort) &&
               mbar_wait(&bars.s_free, j & 1, abort);
          if (!ok) break;
          tc_fence_after();
          issue_qk(j + 1);
        }
        ok = mbar_wait(&bars.p_full, j & 1, abort);
        if (!ok) break;
        tc_fence_after();
        const uint32_t v_addr = smem_u32(smem + Ly::kV0 + (j & 1) * Ly::kTileBytes);
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk) {
          const uint32_t poff = (kk >> 2) * kPanelBytes + (kk & 3) * 32;
          const uint32_t voff = kk * 16 * 128;  // 16 keys x 128-byte rows
          mma_bf16(tO, smem_desc_sw128(p_addr + poff, 16, 1024),
                   smem_desc_sw128(v_addr + voff, kPanelBytes, 1024), idesc_pv,
                   (j > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(&bars.o_done);
        mma_commit(&bars.kv_empty[j & 1]);
      }
      if (!ok) fail();
    }
  } else {
    // ------------------------------------------------------------ softmax warps
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const uint32_t lane_addr = static_cast<uint32_t>(quad * 32) << 16;
    const int node = node0 + r / a.G;
    const int hh = r % a.G;
    const uint32_t* mrow =
        node < a.N ? a.mask + (static_cast<size_t>(b) * a.N + node) * a.W : nullptr;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nt; ++j) {
      if (!mbar_wait(&bars.s_full, j & 1, abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[kBN];
#pragma unroll
      for (int c = 0; c < kBN / 32; ++c)
        tmem_ld32(tS + lane_addr + c * 32, *reinterpret_cast<float(*)[32]>(s + c * 32));
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(&bars.s_free);
      // masks: prefix keys beyond kv_len; tree keys outside the ancestor set
      float mx = -INFINITY;
      if (j < n_prefix) {
        const int lim = kv - (t_begin + j) * kBN;
#pragma unroll
        for (int c = 0; c < kBN; ++c) {
          s[c] = c < lim ? s[c] * a.scale_log2 : -INFINITY;
          mx = fmaxf(mx, s[c]);
        }
      } else {
        const int jt0 = (j - n_prefix) * kBN;
        uint32_t bits[kBN / 32];
#pragma unroll
        for (int w = 0; w < kBN / 32; ++w) {
          const int wi = (jt0 >> 5) + w;
          bits[w] = (mrow && wi < a.W) ? __ldg(mrow + wi) : 0u;
        }
#pragma unroll
        for (int c = 0; c < kBN; ++c) {
          s[c] = ((bits[c >> 5] >> (c & 31)) & 1u) ? s[c] * a.scale_log2 : -INFINITY;
          mx = fmaxf(mx, s[c]);
        }
      }
      const float m_new = fmaxf(m, mx);
      const float m_use = m_new == -INFINITY ? 0.f : m_new;
      const float alpha = m_new == -INFINITY ? 1.f : ex2(m - m_use);
      float rs = 0.f;
#pragma unroll
      for (int c = 0; c < kBN; ++c) {
        s[c] = ex2(s[c] - m_use);
        rs += s[c];
      }
      l = l * alpha + rs;
      m = m_new;
      if (j > 0) {  // P buffer and O are free once PV_{j-1} completed
        if (!mbar_wait(&bars.o_done, (j - 1) & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
      }
      // P row r -> shared memory, bf16, 128-byte swizzle, two 64-key panels
#pragma unroll
      for (int c16 = 0; c16 < kBN / 8; ++c16) {
        uint4 u;
        uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const __nv_bfloat162 v = __floats2bfloat162_rn(s[c16 * 8 + 2 * e], s[c16 * 8 + 2 * e + 1]);
          w[e] = *reinterpret_cast<const uint32_t*>(&v);
        }
        const int panel = c16 >> 3, chunk = c16 & 7;
        *reinterpret_cast<uint4*>(sP + panel * kPanelBytes + r * 128 + ((chunk ^ (r & 7)) << 4)) = u;
      }
      if (j > 0 && __any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          float o[32];
          tmem_ld32(tO + lane_addr + c * 32, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] *= alpha;
          tmem_st32(tO + lane_addr + c * 32, o);
        }
        tmem_wait_st();
      }
      fence_proxy_async();  // make the P stores visible to the tensor core
      tc_fence_before();
      mbar_arrive(&bars.p_full);
    }
    if (ok && !mbar_wait(&bars.o_done, (nt - 1) & 1, abort)) ok = false;
    if (ok) {
      tc_fence_after();
      float o[D];
#pragma unroll
      for (int c = 0; c < D / 32; ++c)
        tmem_ld32(tO + lane_addr + c * 32, *reinterpret_cast<float(*)[32]>(o + c * 32));
      tmem_wait_ld();
      if (a.n_splits == 1) {
        write_row<D>(a, b, g, node, hh, nn, o, m, l);
      } else {
        float* dst = a.ws_o + (static_cast<size_t>(blockIdx.x) * kBM + r) * D;
#pragma unroll
        for (int c = 0; c < D; c += 4)
          *reinterpret_cast<float4*>(dst + c) = make_float4(o[c], o[c + 1], o[c + 2], o[c + 3]);
        a.ws_ml[static_cast<size_t>(blockIdx.x) * kBM + r] = make_float2(m, l);
      }
    } else {
      fail();
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// Merge the KV-split partials of one row: one warp per row, 4 columns per lane.
template <int D>
__global__ void __launch_bounds__(256) combine_kernel(const Args a) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t row_id = static_cast<size_t>(blockIdx.x) * 8 + warp;  // over (b, g, mt, r)
  const int r = static_cast<int>(row_id % kBM);
  size_t idx = row_id / kBM;
  const int mt = static_cast<int>(idx % a.n_mt);
  idx /= a.n_mt;
  const int g = static_cast<int>(idx % a.Hkv);
  const int b = static_cast<int>(idx / a.Hkv);
  if (b >= a.B) return;
  const int node = mt * (kBM / a.G) + r / a.G, hh = r % a.G;
  if (node >= a.N) return;
  int nn = a.n_nodes[b];
  if (nn < 0 || nn > a.N) nn = nn < 0 ? 0 : a.N;
  const size_t cta0 = ((static_cast<size_t>(b) * a.Hkv + g) * a.n_mt + mt) * a.n_splits;
  float M = -INFINITY;
  for (int s = 0; s < a.n_splits; ++s) M = fmaxf(M, a.ws_ml[(cta0 + s) * kBM + r].x);
  constexpr int kPer = D / 32;
  float acc[kPer] = {};
  float Lsum = 0.f;
  if (M != -INFINITY) {
    for (int s = 0; s < a.n_splits; ++s) {
      const float2 ml = a.ws_ml[(cta0 + s) * kBM + r];
      if (ml.x == -INFINITY) continue;
      const float w = ex2(ml.x - M);
      Lsum += ml.y * w;
      const float* src = a.ws_o + ((cta0 + s) * kBM + r) * D + lane * kPer;
#pragma unroll
      for (int e = 0; e < kPer; ++e) acc[e] += w * src[e];
    }
  }
  const int h = g * a.G + hh;
  const bool used = node < nn && Lsum > 0.f;
  const float inv = used ? 1.f / Lsum : 0.f;
  __nv_bfloat16* dst = a.out + ((static_cast<size_t>(b) * a.N + node) * a.Hq + h) * D + lane * kPer;
#pragma unroll
  for (int e = 0; e < kPer; e += 2)
    *reinterpret_cast<__nv_bfloat162*>(dst + e) = __floats2bfloat162_rn(acc[e] * inv, acc[e + 1] * inv);
  if (lane == 0 && a.lse)
    a.lse[(static_cast<size_t>(b) * a.N + node) * a.Hq + h] =
        used ? (M + log2f(Lsum)) * kLn2 : -INFINITY;
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
  int G, n_mt, n_splits;
  size_t ctas;
};

Plan make_plan(int B, int N, int Hq, int Hkv, int Tmax) {
  Plan p;
  p.G = Hq / Hkv;
  p.n_mt = (N * p.G + kBM - 1) / kBM;
  const long long units = static_cast<long long>(B) * Hkv * p.n_mt;
  const int prefix_tiles = (Tmax + kBN - 1) / kBN;
  const int max_splits = prefix_tiles / 4 > 1 ? prefix_tiles / 4 : 1;
  const int sms = sm_count();
  // Pick the split count with the best wave quantisation, lightly penalising splits.
  int best = 1;
  double best_cost = 1e30;
  for (int s = 1; s <= max_splits && s <= 64; ++s) {
    const double ctas = static_cast<double>(units) * s;
    const double waves = std::ceil(ctas / sms);
    const double work = (prefix_tiles + 1.0) / s + 1.0;  // tiles per CTA + fixed cost
    const double cost = waves * work * (1.0 + 0.01 * s);
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best = s;
    }
  }
  p.n_splits = best;
  p.ctas = static_cast<size_t>(units) * p.n_splits;
  return p;
}

size_t ws_layout(const Plan& p, int D, char* base, float** o, float2** ml) {
  if (p.n_splits == 1) return 256;
  const size_t ob = align_up(p.ctas * kBM * D * sizeof(float), 256);
  const size_t mb = align_up(p.ctas * kBM * sizeof(float2), 256);
  if (base) {
    *o = reinterpret_cast<float*>(base);
    *ml = reinterpret_cast<float2*>(base + ob);
  }
  return ob + mb;
}

template <int D>
void set_smem_attr() {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         Layout<D>::kAlloc);
  });
}

}  // namespace
}  // namespace presto

using namespace presto;

extern "C" size_t presto_attn_workspace(int B, int N, int Hq, int Hkv, int D, int Tmax) {
  if (B < 1 || N < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv || Tmax < 0 || (D != 64 && D != 128))
    return 0;
  return ws_layout(make_plan(B, N, Hq, Hkv, Tmax), D, nullptr, nullptr, nullptr);
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
  const Plan p = make_plan(B, N, Hq, Hkv, Tmax);
  Args a{};
  if (p.n_splits > 1) {
    if (!ws || reinterpret_cast<uintptr_t>(ws) % 256 ||
        ws_bytes < ws_layout(p, D, nullptr, nullptr, nullptr))
      return PRESTO_ERR_WORKSPACE;
    ws_layout(p, D, static_cast<char*>(ws), &a.ws_o, &a.ws_ml);
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
  const dim3 grid(static_cast<unsigned>(p.ctas));
  if (D == 128) {
    set_smem_attr<128>();
    attn_kernel<128><<<grid, kThreads, Layout<128>::kAlloc, stream>>>(tq, tkc, tvc, tkt, tvt, a);
  } else {
    set_smem_attr<64>();
    attn_kernel<64><<<grid, kThreads, Layout<64>::kAlloc, stream>>>(tq, tkc, tvc, tkt, tvt, a);
  }
  if (cudaGetLastError() != cudaSuccess) return PRESTO_ERR_CUDA;
  if (p.n_splits > 1) {
    const size_t rows = static_cast<size_t>(B) * Hkv * p.n_mt * kBM;
    const unsigned blocks = static_cast<unsigned>((rows + 7) / 8);
    if (D == 128)
      combine_kernel<128><<<blocks, 256, 0, stream>>>(a);
    else
      combine_kernel<64><<<blocks, 256, 0, stream>>>(a);
  }
  return launch_status();
}
