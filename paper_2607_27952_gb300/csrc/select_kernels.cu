// Host side of the selection (Eq. 9-12): kernel variant, cluster size, tensor
// map and launch.  The kernel itself is in select_impl.cuh; its instantiations
// are in select_f32.cu, select_bf16.cu and select_bf16_tc.cu.
#include "select_impl.cuh"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <map>
#include <mutex>
#include <tuple>

namespace last {

void *select_pick_f32(int nch);
void *select_pick_bf16(int nch, int tb);
void *select_pick_bf16_tc(int nch);

namespace {

void *pick_select(int dtype, int nch, int tb, bool tc) {
  // fp32 rows take twice the registers per prefetched group: 2-token blocks only;
  // the tensor-core update exists for bf16 (its CUDA-core block width is unused)
  if (dtype != LAST_DTYPE_BF16) return select_pick_f32(nch);
  if (tc) return select_pick_bf16_tc(nch);
  return select_pick_bf16(nch, tb);
}

struct DeviceInfo {
  int optin = 0, sms = 0;
  double l2 = 0.0;
  double dram_bytes_per_cycle = 0.0;   // sustained DRAM bytes per SM clock, whole device
};
// Queried once per device: some attributes (clock rates) are slow to read.
DeviceInfo device_info() {
  static std::mutex mu;
  static std::map<int, DeviceInfo> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  {
    std::lock_guard<std::mutex> lock(mu);
    auto hit = cache.find(dev);
    if (hit != cache.end()) return hit->second;
  }
  DeviceInfo d;
  int v = 0, mem_khz = 0, bus_bits = 0, sm_khz = 0;
  cudaDeviceGetAttribute(&d.optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&v, cudaDevAttrL2CacheSize, dev);
  cudaDeviceGetAttribute(&mem_khz, cudaDevAttrMemoryClockRate, dev);
  cudaDeviceGetAttribute(&bus_bits, cudaDevAttrGlobalMemoryBusWidth, dev);
  cudaDeviceGetAttribute(&sm_khz, cudaDevAttrClockRate, dev);
  d.l2 = v;
  // double data rate; about 80% of the nominal rate is sustained
  if (mem_khz > 0 && bus_bits > 0 && sm_khz > 0)
    d.dram_bytes_per_cycle = 0.8 * 2.0 * mem_khz * (bus_bits / 8.0) / sm_khz;
  else
    d.dram_bytes_per_cycle = 3000.0;
  std::lock_guard<std::mutex> lock(mu);
  cache.emplace(dev, d);
  return d;
}

// Clusters of `fn` (csize CTAs, smem bytes each) resident at once, cached per
// (device, kernel, cluster size, shared memory); 0 if it cannot be placed.
int active_clusters(void *fn, int csize, size_t smem) {
  static std::mutex mu;
  static std::map<std::tuple<int, void *, int, size_t>, int> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  const auto key = std::make_tuple(dev, fn, csize, smem);
  {
    std::lock_guard<std::mutex> lock(mu);
    auto hit = cache.find(key);
    if (hit != cache.end()) return hit->second;
  }
  int active = 0;
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess &&
      cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) == cudaSuccess) {
    cudaLaunchConfig_t q = {};
    q.gridDim = dim3(csize);
    q.blockDim = dim3(kSelThreads);
    q.dynamicSmemBytes = smem;
    cudaLaunchAttribute qa[1];
    qa[0].id = cudaLaunchAttributeClusterDimension;
    qa[0].val.clusterDim.x = csize;
    qa[0].val.clusterDim.y = 1;
    qa[0].val.clusterDim.z = 1;
    q.attrs = qa;
    q.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&active, fn, &q) != cudaSuccess) active = 0;
  }
  cudaGetLastError();
  std::lock_guard<std::mutex> lock(mu);
  cache.emplace(key, active);
  return active;
}

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link-time
// dependency on the driver library); nullptr if unavailable.
EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = []() -> EncodeTiledFn {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    return reinterpret_cast<EncodeTiledFn>(p);
  }();
  return fn;
}

// X as a [rows][dv] bf16 tensor, 64-element x box_rows boxes, 128-byte swizzle.
bool encode_x_map(CUtensorMap *m, const void *x, long long rows, int dv, int box_rows = kTcBM) {
  EncodeTiledFn fn = encode_tiled();
  if (fn == nullptr || rows <= 0) return false;
  cuuint64_t dims[2] = {(cuuint64_t)dv, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)dv * 2};
  cuuint32_t box[2] = {(cuuint32_t)kTcBK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(x), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Bytes of feature rows a CTA streams in one dense update below which the
// selection does not skip rows by the triangle inequality.
constexpr double kTriMinStreamBytes = 2.0 * 1024 * 1024;
// the selection keeps each token's nearest root id in 16 bits
static_assert(kMaxRoots <= 32767, "root ids must fit int16_t");

// Opt-in shared memory per CTA of the sm_100 class, for checks made before a
// device is at hand.
constexpr int kSmemOptinSm100 = 232448;

// Token block width of the kernel variant (the shared-memory plan depends on it):
// 2 for fp32 and the tensor-core update, else 4 unless a CTA owns few tokens.
int select_tb(int elem, bool tc, int tpc_max) { return (elem == 4 || tc || tpc_max < 64) ? 2 : 4; }

}  // namespace

bool select_supported(const Plan &pl, std::string *why) {
  if (pl.dv < 8 || pl.dv % 8 != 0 || pl.dv > kMaxFeatDim) {
    if (why) *why = "feat_dim must be a positive multiple of 8, at most 2048";
    return false;
  }
  return true;
}

bool select_fits(const Plan &pl, std::string *why) {
  // The largest request: the CUDA-core update's per-token state of one of 16
  // clustered CTAs, with a row ring and no row cache, within sm_100-class shared
  // memory (the launch itself takes the device's own figure).  Past that, up to
  // kGridMaxReq requests run on the whole GPU (select_grid.cu) when their tokens
  // fit its CTAs' shared memory.
  const int tpc = (pl.max_vis + kMaxCluster - 1) / kMaxCluster;
  const int tb = select_tb(pl.elem, false, tpc);
  if (select_smem(0, pl.dv * pl.elem, tpc, 1, tb, pl.elem, kLcap / 2).total > (size_t)kSmemOptinSm100 &&
      !(pl.B <= kGridMaxReq && grid_select_fits(pl))) {
    if (why) *why = "a request has too many visual tokens for the selection's shared-memory plan";
    return false;
  }
  return true;
}

// Bound on |d~ - d| between a tensor-core distance d~ = 1 - (dot~ r_i) r_j and the
// canonical one, in units of cosine distance.  Both dots carry exact bf16 products;
// the canonical order adds each lane's dv/256 * 8 products and five butterfly levels
// (error <= 80 ulp-units of sum |x_i,k x_j,k| <= |x_i||x_j|), and the tensor cores'
// fp32 accumulation is taken at dv * 2^-21 of the same magnitude, 64 times the
// worst error measured on GB300 for dv = 2048 (87 units of 2^-24); the last term
// covers the fp32 roundings of the two scalings and the subtraction.
float tc_distance_eps(int dv) {
  return (float)(((double)dv * std::ldexp(1.0, -21) + 80.0 * std::ldexp(1.0, -24)) * 1.01 + 1e-6);
}

cudaError_t launch_select(const Plan &pl, const float *w, const void *x, int32_t *idx_out,
                          void *x_out, char *ws, cudaStream_t s) {
  if (pl.B == 0 || pl.total_keep == 0) return cudaSuccess;
  const int rb = pl.dv * pl.elem;
  const int nch = (pl.dv + 255) / 256;
  const DeviceInfo di = device_info();
  SelectArgs a;
  std::memset(&a, 0, sizeof a);
  // bf16 rows take the tensor-core update when the X tensor map can be encoded
  bool tc = pl.dtype == LAST_DTYPE_BF16 && encode_x_map(&a.tmap, x, pl.total_vis, pl.dv);

  // Cluster size: every size the device can place is costed as
  //   waves x (one round's update + round overhead)
  // (the round count of a request does not depend on C to first order); small
  // clusters raise the number of requests in flight, large ones shorten each round.
  // When no cluster size fits the tensor-core update (its accumulators take a
  // TMEM column per list entry and 128-row tile, so very long requests do not
  // fit), the sizes are costed again for the CUDA-core update.
  int C = 0, tpc = 0, cache_rows = 0, ring = 0, lcap = kLcap / 2, stages = 0, kps = 1, roots = 0;
  int gram = 0;
  size_t smem = 0;
  double best = 0.0;
  void *fn = nullptr;
  for (int pass = 0; pass < 2 && C == 0; ++pass) {
  if (pass == 1) {
    if (!tc) break;
    tc = false;
  }
  for (int c = 1; c <= kMaxCluster; c = tc ? c + 1 : 2 * c) {
    const int tpc_c = (pl.max_vis + c - 1) / c;
    const int tb_c = select_tb(pl.elem, tc, tpc_c);
    void *fn_c = pick_select(pl.dtype, nch, tb_c, tc);
    int cache_c = 0, ring_c = 0, lcap_c = 0, stages_c = 0, kps_c = 1, roots_c = 0, gram_c = 0;
    size_t smem_c = 0;
    if (tc) {
      // the list length is the MMA N: lcap accumulator columns per 128-row tile; the
      // TMA ring takes the shared memory left over
      const int tiles = (tpc_c + kTcBM - 1) / kTcBM;
      // stages of kps boxes: the largest kps (<= 4) that still leaves 2 stages.  A list
      // of kLcap entries is tried first (it accepts more picks per round), then half.
      for (int lc = kLcap; lc >= kLcap / 2 && lcap_c == 0; lc /= 2) {
        // Row skipping: a CTA's slice of the roots is the M = 128 operand of its
        // root-table MMA, so the request's roots are capped at 128 per CTA.  It is
        // used only where a CTA's dense update streams at least kTriMinStreamBytes:
        // below that the per-round root table costs about what it saves (measured on
        // 576-token requests in clusters of two).
        const bool tri_c = pl.root_rows > 0 && (double)tpc_c * rb >= kTriMinStreamBytes;
        const int roots_lc = tri_c ? std::min(kMaxRoots, kTcBM * c) : 0;
        // the list's Gram only when the pair dots would take more than two passes of
        // the cluster's pair workers (at least six warps per CTA)
        const int gram_lc = lc * (lc - 1) / 2 > 2 * c * (kSelectWarps - 2) * 4 ? 1 : 0;
        const size_t fixed = select_smem(0, rb, tpc_c, 0, tb_c, pl.elem, lc, 1, 0, 1, roots_lc, c,
                                         gram_lc).total;
        // TMEM: lc columns per tile plus kGramChains x lc for the list's Gram
        if (fixed + 2 * (size_t)kTcBoxBytes > (size_t)di.optin ||
            (tiles + kGramChains) * lc > kTmemCols)
          continue;
        const size_t room = di.optin - fixed;
        kps_c = 1;
        while (kps_c < 4 && room >= 2 * (size_t)(2 * kps_c) * kTcBoxBytes) kps_c *= 2;
        kps_c = std::min(kps_c, tc_kblocks(pl.dv));
        stages_c = (int)std::min<size_t>(kTcMaxStages, room / ((size_t)kps_c * kTcBoxBytes));
        lcap_c = lc;
        roots_c = roots_lc;
        gram_c = gram_lc;
        smem_c = select_smem(0, rb, tpc_c, 0, tb_c, pl.elem, lc, 1, stages_c, kps_c, roots_c, c,
                             gram_c).total;
      }
      if (lcap_c == 0) continue;
    } else {
      lcap_c = c <= 4 ? kLcap : kLcap / 2;
      // rows that fit without a ring; otherwise reserve the ring and cache what is left
      const size_t fixed0 = select_smem(0, rb, tpc_c, 0, tb_c, pl.elem, lcap_c, 0, 0, 1, 0, c).total;
      if (fixed0 > (size_t)di.optin) continue;
      cache_c = (int)std::min<size_t>(tpc_c, (di.optin - fixed0) / rb);
      if (cache_c < tpc_c) {
        ring_c = 1;
        const size_t fixed1 = select_smem(0, rb, tpc_c, 1, tb_c, pl.elem, lcap_c, 0, 0, 1, 0, c).total;
        if (fixed1 > (size_t)di.optin) continue;
        cache_c = (int)std::min<size_t>(tpc_c, (di.optin - fixed1) / rb);
      }
      smem_c = select_smem(cache_c, rb, tpc_c, ring_c, tb_c, pl.elem, lcap_c, 0, 0, 1, 0, c).total;
    }
    const int active = active_clusters(fn_c, c, smem_c);
    if (active <= 0) continue;
    const double waves = std::ceil((double)pl.B / active);
    // features of the requests in flight beyond L2 stream from HBM
    const double in_flight = std::min<double>(pl.B, active) * pl.max_vis * (double)rb;
    const bool from_hbm = in_flight > 0.7 * di.l2;
    double round_cycles;
    if (tc) {
      // The update streams this CTA's rows (whole 128-row tiles) once per round, at
      // the smallest of the ring's hand-off rate (about 900 cycles per stage), the
      // rate one SM's TMA sustains (about 26 bytes per clock; both measured on
      // GB300) and this CTA's share of DRAM (or of L2, taken as 2.5x, when the
      // features of the requests in flight fit in it).
      const double bytes = (double)((tpc_c + kTcBM - 1) / kTcBM) * kTcBM * tc_kblocks(pl.dv) * 128.0;
      const double ctas = std::min<double>(pl.B, active) * c;
      const double share = di.dram_bytes_per_cycle / ctas * (from_hbm ? 1.0 : 2.5);
      const double bw = std::min(std::min(kps_c * (double)kTcBoxBytes / 900.0, 26.0), share);
      round_cycles = bytes / bw + 30000.0 + 400.0 * c;
      // a 16-entry list accepts fewer consecutive picks per round than a 32-entry
      // one: a host replay of the rounds on the benchmark presets needs 1.4-1.6x the
      // rounds (c3, c4 and the video batch), so its rounds are weighted by 1.4
      if (lcap_c < kLcap) round_cycles *= 1.4;
    } else {
      const double stream_penalty = from_hbm ? 3.0 : 1.0;
      const double streamed = std::max(0, tpc_c - cache_c), cached = std::min(tpc_c, cache_c);
      round_cycles = (cached + stream_penalty * streamed) * pl.dv * 8.0 / 56.0 + 16000.0 + 400.0 * c;
    }
    const double cost = waves * round_cycles;
    if (C == 0 || cost < best) {
      best = cost; C = c; tpc = tpc_c; cache_rows = cache_c; smem = smem_c; ring = ring_c;
      lcap = lcap_c; fn = fn_c; stages = stages_c; kps = kps_c; roots = roots_c; gram = gram_c;
    }
  }
  }
  if (C == 0) {
    // requests too long for any cluster: up to kGridMaxReq of them on the whole GPU
    if (pl.B <= kGridMaxReq && grid_select_fits(pl))
      return launch_select_grid(pl, w, x, idx_out, x_out, ws, s);
    return cudaErrorInvalidConfiguration;
  }
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;

  a.x = x; a.w = w; a.idx_out = idx_out; a.x_out = x_out;
  a.meta = reinterpret_cast<const int32_t *>(ws + pl.off_meta);
  a.order = reinterpret_cast<const int32_t *>(ws + pl.off_order);
  a.dv = pl.dv; a.row_bytes = rb; a.tpc_max = tpc; a.cache_rows = cache_rows; a.csize = C;
  // Candidates each CTA publishes (the cluster's list is a C-way merge of the
  // published lists, so its cost does not grow with them).  The tensor-core variant
  // publishes its top 16 (its incremental candidate list holds them cheaply) and
  // accepts up to 32 picks a round; the CUDA-core update ranks 8 (4 in clusters of
  // more than 4 CTAs) and accepts 16 (its register blocking).
  if (tc) {
    a.mc = kTopMax - 1;   // the candidate list keeps every CTA's top keys cheaply
    a.max_accept = kMaxAccept;
  } else {
    a.mc = C <= 4 ? 8 : 4;
    a.max_accept = 16;
  }
  a.ring = ring;
  a.lcap = lcap;
  a.gram = gram;
  a.err = reinterpret_cast<unsigned *>(ws + pl.off_err);
  if (tc) {
    const int cols = ((tpc + kTcBM - 1) / kTcBM + kGramChains) * lcap;   // tiles + the list Gram
    uint32_t tcols = 32;
    while ((int)tcols < cols) tcols *= 2;
    a.tmem_cols = tcols;
    a.tc_stages = stages;
    a.tc_kps = kps;
    a.tc_eps = tc_distance_eps(pl.dv);
    // row skipping (the root capacity was chosen with the shared-memory plan)
    if (roots > 0) {
      a.tri = 1;
      a.root_cap = roots;
      a.roots = ws + pl.off_roots;
      a.rtab = reinterpret_cast<float *>(ws + pl.off_rtab);
      a.tri_eps_x = a.tc_eps + kTriEpsC;
    }
  }

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(C * pl.B);
  cfg.blockDim = dim3(kSelThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void *args[] = {&a};
  return cudaLaunchKernelExC(&cfg, fn, args);
}

}  // namespace last
