// presto_tree_mask (§4.3, App. C (I), (IV): each draft token attends to its
// ancestors) and presto_accept (§2.1 greedy prefix acceptance, App. A alpha_T(P),
// App. C (I) bonus token).
#include "common.cuh"

namespace presto {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kMaxW = kMaxN / 32;

// One CTA per sequence, one thread per node: walk the parent chain (at most L
// steps, parents in shared memory) and set one bit per ancestor-or-self.
__global__ void __launch_bounds__(kMaxN) mask_kernel(const int32_t* node_parent,
                                                     const int32_t* node_depth,
                                                     const int32_t* n_nodes,
                                                     const int32_t* kv_len, int N, int W,
                                                     uint32_t* mask, int32_t* pos_ids,
                                                     int32_t* dev_status) {
  __shared__ int par[kMaxN];
  __shared__ int dep[kMaxN];
  extern __shared__ uint32_t rows[];  // [N][W + 1]
  pdl_launch_dependents();
  pdl_wait();  // the tree comes from the previous kernel on the stream
  const int b = blockIdx.x, i = threadIdx.x;
  int n = n_nodes[b];
  if (n < 1 || n > N) {
    if (i == 0) report(dev_status, PRESTO_DEV_BAD_NNODES);
    n = n < 1 ? 0 : N;
  }
  const int kv = kv_len[b];
  if (i == 0 && kv < 0) report(dev_status, PRESTO_DEV_BAD_KVLEN);
  if (i < N) {
    par[i] = node_parent[static_cast<size_t>(b) * N + i];
    dep[i] = node_depth[static_cast<size_t>(b) * N + i];
    for (int w = 0; w < W; ++w) rows[i * (W + 1) + w] = 0u;
  }
  __syncthreads();
  if (i < n) {
    bool bad = (i == 0) ? (par[0] != -1 || dep[0] != 0)
                        : (par[i] < 0 || par[i] >= i || dep[i] != dep[par[i]] + 1);
    // parents strictly decrease, so the walk ends within i steps
    int j = i;
    for (;;) {
      rows[i * (W + 1) + (j >> 5)] |= 1u << (j & 31);
      if (j == 0) break;
      const int p = par[j];
      if (p < 0 || p >= j) {
        bad = true;
        break;
      }
      j = p;
    }
    if (bad) report(dev_status, PRESTO_DEV_BAD_PARENT);
  }
  __syncthreads();
  for (int e = i; e < N * W; e += blockDim.x) {
    const int r = e / W, w = e % W;
    mask[static_cast<size_t>(b) * N * W + e] = rows[r * (W + 1) + w];
  }
  if (i < N) pos_ids[static_cast<size_t>(b) * N + i] = i < n ? kv + dep[i] : -1;
}

// One warp per sequence.  match(i) = (i == 0) || token(i) == target(parent(i));
// node i is accepted iff every node of its mask row matches; the deepest accepted
// node (unique when siblings carry distinct tokens; lowest index otherwise) ends
// the path, whose nodes are the set bits of its mask row in index order.
__global__ void __launch_bounds__(32) accept_kernel(
    const int32_t* node_token, const int32_t* node_parent, const int32_t* node_depth,
    const uint32_t* mask, const int32_t* n_nodes, const int32_t* target_token, int N, int W,
    int L, int32_t* accept_len, int32_t* accept_path, int32_t* bonus, int32_t* dev_status) {
  pdl_launch_dependents();
  pdl_wait();  // the tree and the target tokens come from earlier kernels on the stream
  const int b = blockIdx.x, lane = threadIdx.x;
  int n = n_nodes[b];
  if (n < 1 || n > N) {
    if (lane == 0) report(dev_status, PRESTO_DEV_BAD_NNODES);
    n = n < 1 ? 1 : N;
  }
  const size_t base = static_cast<size_t>(b) * N;
  __shared__ uint32_t matched[kMaxW];
  for (int w = 0; w < W; ++w) {
    const int i = w * 32 + lane;
    bool m = false;
    if (i < n) {
      if (i == 0) {
        m = true;
      } else {
        const int p = node_parent[base + i];
        if (p >= 0 && p < i)
          m = node_token[base + i] == target_token[base + p];
        else
          report(dev_status, PRESTO_DEV_BAD_PARENT);
      }
    }
    const uint32_t bal = __ballot_sync(kFull, m);
    if (lane == 0) matched[w] = bal;
  }
  __syncwarp();
  // deepest accepted node: maximise (depth, -index)
  unsigned bestkey = 0u;
  for (int w = 0; w < W; ++w) {
    const int i = w * 32 + lane;
    if (i < n) {
      const uint32_t* row = mask + (base + i) * W;
      bool ok = true;
      for (int u = 0; u < W; ++u) ok &= (row[u] & ~matched[u]) == 0u;
      if (ok) {
        const int d = node_depth[base + i];
        const unsigned key = (static_cast<unsigned>(d & 0x3F) << 10) | (1023u - i);
        bestkey = bestkey > key ? bestkey : key;
      }
    }
  }
  const unsigned top = __reduce_max_sync(kFull, bestkey);
  const int best = 1023 - static_cast<int>(top & 1023u);
  const uint32_t* row = mask + (base + best) * W;
  // path: set bits of the row in increasing index order, written by prefix count
  int written = 0;
  for (int u = 0; u < W; ++u) {
    const uint32_t bits = row[u];
    const int i = u * 32 + lane;
    if ((bits >> lane) & 1u) {
      const int slot = written + __popc(bits & ((1u << lane) - 1u));
      if (slot <= L) accept_path[static_cast<size_t>(b) * (L + 1) + slot] = i;
    }
    written += __popc(bits);
  }
  for (int s = written + lane; s <= L; s += 32) accept_path[static_cast<size_t>(b) * (L + 1) + s] = -1;
  if (lane == 0) {
    if (written > L + 1) report(dev_status, PRESTO_DEV_BAD_PARENT);
    accept_len[b] = node_depth[base + best];
    bonus[b] = target_token[base + best];
  }
}

}  // namespace
}  // namespace presto

using namespace presto;

extern "C" int presto_tree_mask(const int32_t* node_parent, const int32_t* node_depth,
                                const int32_t* n_nodes, const int32_t* kv_len, int B, int N,
                                uint32_t* mask, int32_t* pos_ids, int32_t* dev_status,
                                presto_stream_t stream) {
  PRESTO_CHECK_ARG(node_parent && node_depth && n_nodes && kv_len && mask && pos_ids);
  PRESTO_CHECK_ARG(B >= 1 && N >= 1);
  PRESTO_CHECK_LIMIT(N <= kMaxN);
  const int W = (N + 31) / 32;
  const int threads = (N + 31) / 32 * 32;
  cudaLaunchConfig_t cfg{};
  const size_t rows_bytes = static_cast<size_t>(N) * (W + 1) * 4;
  static const cudaError_t attr_ok = cudaFuncSetAttribute(
      mask_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
      static_cast<int>(static_cast<size_t>(kMaxN) * (kMaxN / 32 + 1) * 4));
  if (attr_ok != cudaSuccess) return PRESTO_ERR_CUDA;
  cfg.gridDim = dim3(static_cast<unsigned>(B));
  cfg.blockDim = dim3(static_cast<unsigned>(threads));
  cfg.dynamicSmemBytes = rows_bytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1] = {pdl_attribute()};
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, mask_kernel, node_parent, node_depth, n_nodes, kv_len, N, W, mask,
                         pos_ids, dev_status) != cudaSuccess)
    return PRESTO_ERR_CUDA;
  return launch_status();
}

extern "C" int presto_accept(const int32_t* node_token, const int32_t* node_parent,
                             const int32_t* node_depth, const uint32_t* mask,
                             const int32_t* n_nodes, const int32_t* target_token, int B, int N,
                             int L, int32_t* accept_len, int32_t* accept_path, int32_t* bonus,
                             int32_t* dev_status, presto_stream_t stream) {
  PRESTO_CHECK_ARG(node_token && node_parent && node_depth && mask && n_nodes && target_token &&
                   accept_len && accept_path && bonus);
  PRESTO_CHECK_ARG(B >= 1 && N >= 1 && L >= 1);
  PRESTO_CHECK_LIMIT(N <= kMaxN && L <= kMaxL);
  const int W = (N + 31) / 32;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(B));
  cfg.blockDim = dim3(32);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1] = {pdl_attribute()};
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, accept_kernel, node_token, node_parent, node_depth, mask, n_nodes,
                         target_token, N, W, L, accept_len, accept_path, bonus,
                         dev_status) != cudaSuccess)
    return PRESTO_ERR_CUDA;
  return launch_status();
}
