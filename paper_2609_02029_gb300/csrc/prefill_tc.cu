// prefill_tc.cu -- window-limited causal prefill on the 5th-generation tensor
// cores (tcgen05 + TMEM + TMA) (HeadWiseKV Sec. 3.2, Eq. conditional-attention-
// weight and Eq. conditional-attention for every prompt position; Sec. 3.3:
// each KV head reads only its own ring).
//
// Query p in [t0, t0+n) of query head q attends to KV head q/G at positions
// [max(0, p-W+1), p]: positions < t0 from the head's ring, >= t0 from the
// chunk's own K/V. The ring is walked in slot order (slot j holds the unique
// retained position congruent to j mod cap), so wrap needs no special case;
// each key column carries its position and the window/causal mask is applied
// per element on the tiles that need it. Tiles no row of the block can see are
// never loaded, so a short-window head does window-sized work.
//
// CTA = one 128-row query tile: 128/G positions x the G query heads of one KV
// head (the GQA group shares every K/V tile). Warp roles:
//   warp 0      TMA producer: Q once, then K/V tiles into a STAGES-deep ring
//   warp 1      MMA issuer (one thread): S = Q K^T into a double-buffered TMEM
//               tile (128 x BN fp32), then O += P V into TMEM (128 x D fp32)
//   warps 2+    softmax: thread r owns TMEM lane r = query row r, so the row
//               max and sum are thread-local (at head_dim <= 128 two warps
//               share each row quarter, splitting its columns and exchanging
//               the row max through shared memory); P goes back to TMEM as bf16
//               and is the tensor-memory A operand of the PV mma; O is rescaled in TMEM only
//               when a row's running max grows by more than 2^8 (the final
//               O / l uses the same reference, so the result is exact).
// While the softmax warps work on tile j the tensor core computes S of tile j+1.
// All waits are bounded; a thread that gives up stops waiting and issuing but
// keeps walking the tile sequence, so every role reaches the TMEM release.
#include "hwkv_internal.cuh"

namespace hwkv {

namespace {

template <int D, int BN, int STAGES, int SPLIT, int SBUF = 2, int CTAS = 1>
struct TcCfg {
  static constexpr int kSBuf = SBUF;          // S buffers in TMEM
  static constexpr int kCtasPerSm = CTAS;     // resident CTAs per SM (registers, TMEM, smem)
  static constexpr int kSoftmaxWarps = 4 * SPLIT;  // SPLIT warps share each TMEM lane quarter
  static constexpr int kThreads = 64 + 32 * kSoftmaxWarps;
  static constexpr int kCW = BN / SPLIT;           // S columns per softmax warp
  static constexpr int kOW = D / SPLIT;            // O columns per softmax warp
  static_assert(kCW % 32 == 0 && kOW % 32 == 0, "column split");
  static constexpr int kSlabs = D / 64;
  static constexpr int kQSlab = 128 * 128;             // 128 rows x 128 B
  static constexpr int kQBytes = kSlabs * kQSlab;
  static constexpr int kKVSlab = BN * 128;             // BN rows x 128 B
  static constexpr int kTileBytes = kSlabs * kKVSlab;  // one K (or V) tile
  static constexpr int kStageBytes = 2 * kTileBytes;
  // TMEM columns: S0 [0, BN), S1 [BN, 2BN), O [2BN, 2BN + D), P [2BN + D, 2BN + D + BN/2)
  static constexpr int kColO = SBUF * BN;
  static constexpr int kColP = SBUF * BN + D;
  static constexpr int kBarBytes = 256;
  static constexpr int kRedBytes = SPLIT > 1 ? 2 * 2 * 128 * 4 : 0;  // row-max exchange
  static constexpr int kSmem =
      kQBytes + STAGES * kStageBytes + kBarBytes + kRedBytes + 1024;
  static constexpr int kTmemNeed = SBUF * BN + D + BN / 2;
  static constexpr uint32_t kTmemCols = kTmemNeed <= 128 ? 128 : (kTmemNeed <= 256 ? 256 : 512);
  static_assert(kTmemCols * CTAS <= 512, "TMEM: S buffers, O and P of every resident CTA");
};

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int32_t x,
                                            int32_t y, int32_t z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

// The key tiles one query block needs, in order: the sink slots (all read by
// every row), then tiles of the window region (slots S .. cap-1, positions >= S,
// position p in slot S + (p - S) mod Wr) whose newest held position reaches the
// block's lowest visible key, then chunk tiles up to the block's last row (from
// the chunk's start while it still holds sink positions). A ring tile's j0 is its
// first ring slot. Every role walks the same sequence. Without sinks (S = 0) the
// window region is the whole ring.
template <int BN>
struct KeySeq {
  int64_t t0, n, W, S, Wr, n_sink, tw, n_win, r0, lo_need, c_first, n_chunk_tiles;
  int64_t n_sink_tiles, n_win_tiles;
  bool win_needed;
  int64_t sink_cur, win_cur, chunk_cur;

  __device__ void init(const PrefillUnit& u, int64_t t0_, int64_t n_, int64_t p0, int64_t p_last) {
    t0 = t0_;
    n = n_;
    W = u.window;
    S = u.sink;
    Wr = u.cap - S;
    n_sink = t0 < S ? t0 : S;
    tw = t0 > S ? t0 - S : 0;            // history tokens in the window region
    n_win = tw < Wr ? tw : Wr;
    r0 = tw % Wr;
    lo_need = W == 0 ? 0 : (p0 - W + 1 > 0 ? p0 - W + 1 : 0);
    n_sink_tiles = (n_sink + BN - 1) / BN;
    n_win_tiles = (n_win + BN - 1) / BN;
    // chunk keys below S are sinks, read by every row
    const int64_t c_lo = t0 < S ? 0 : (t0 > lo_need ? t0 : lo_need) - t0;
    c_first = (c_lo / BN) * BN;
    const int64_t c_hi = p_last - t0;
    n_chunk_tiles = c_hi >= c_first ? (c_hi - c_first) / BN + 1 : 0;
    win_needed = n_win > 0 && (W == 0 || p0 - W + 1 < t0);
    sink_cur = 0;
    win_cur = next_win(0);
    chunk_cur = 0;
  }
  // position held by window-region slot j (0-based within the region)
  __device__ int64_t slot_pos(int64_t j) const {
    if (tw <= Wr) return S + j;
    return S + (j < r0 ? tw - r0 + j : tw - r0 - Wr + j);
  }
  // largest position held in window-region slots [j0, j1] (j1 < n_win)
  __device__ int64_t tile_max_pos(int64_t j0, int64_t j1) const {
    if (tw > Wr && j0 < r0 && r0 <= j1) return slot_pos(r0 - 1);
    return slot_pos(j1);
  }
  __device__ bool win_tile_needed(int64_t jt) const {
    if (!win_needed) return false;
    if (W == 0) return true;
    const int64_t j0 = jt * BN;
    const int64_t j1 = (j0 + BN < n_win ? j0 + BN : n_win) - 1;
    return tile_max_pos(j0, j1) >= lo_need;
  }
  __device__ int64_t next_win(int64_t jt) const {
    for (; jt < n_win_tiles; ++jt)
      if (win_tile_needed(jt)) return jt;
    return -1;
  }
  // hist: 0 = chunk tile, 1 = window-region tile, 2 = sink tile
  __device__ bool next(int& hist, int64_t& j0) {
    if (sink_cur < n_sink_tiles) {
      hist = 2;
      j0 = sink_cur * BN;
      ++sink_cur;
      return true;
    }
    if (win_cur >= 0) {
      hist = 1;
      j0 = S + win_cur * BN;
      win_cur = next_win(win_cur + 1);
      return true;
    }
    if (chunk_cur < n_chunk_tiles) {
      hist = 0;
      j0 = c_first + chunk_cur * BN;
      ++chunk_cur;
      return true;
    }
    return false;
  }
};

__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, int* err,
                                              bool& aborted) {
  if (aborted) return false;
  if (!mbar_wait_bounded(bar, parity, err)) aborted = true;
  return !aborted;
}

// one lane of the warp waits, the warp then proceeds together; the abort flag
// is shared by the warp so every lane takes the same path
__device__ __forceinline__ bool warp_wait_or_abort(uint64_t* bar, uint32_t parity, int* err,
                                                   bool& aborted) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = wait_or_abort(bar, parity, err, aborted) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  aborted = ok == 0;
  return ok != 0;
}

}  // namespace

template <int D, int BN, int STAGES, int SPLIT, int SBUF, int CTAS>
__global__ void __launch_bounds__(TcCfg<D, BN, STAGES, SPLIT, SBUF, CTAS>::kThreads, CTAS)
    prefill_tc_kernel(const __grid_constant__ CUtensorMap q_map,
                      const __grid_constant__ CUtensorMap ck_map,
                      const __grid_constant__ CUtensorMap cv_map,
                      const __grid_constant__ CUtensorMap ring_map, const PrefillParams p) {
  using C = TcCfg<D, BN, STAGES, SPLIT, SBUF, CTAS>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  // K and V tiles live in separate buffers, released separately: a K buffer as soon
  // as its QK^T is done, a V buffer when its PV is done, so the next K tiles load
  // while this tile's softmax and PV run
  uint8_t* sQ = smem;
  uint8_t* sK = smem + C::kQBytes;                      // [STAGES] K tiles
  uint8_t* sV = sK + STAGES * C::kTileBytes;            // [STAGES] V tiles
  uint64_t* bars = reinterpret_cast<uint64_t*>(sK + STAGES * C::kStageBytes);
  uint64_t* k_full = bars;                // [STAGES] K tile landed
  uint64_t* k_empty = bars + STAGES;      // [STAGES] QK^T of that tile done
  uint64_t* v_full = bars + 2 * STAGES;   // [STAGES] V tile landed
  uint64_t* v_empty = bars + 3 * STAGES;  // [STAGES] PV of that tile done
  uint64_t* s_full = bars + 4 * STAGES;   // [2] S tile computed
  uint64_t* s_free = s_full + 2;         // [2] S tile read by the softmax warps
  uint64_t* p_full = s_free + 2;         // P of the current tile written (and O rescaled)
  uint64_t* pv_done = p_full + 1;        // PV mma of the previous tile done
  uint64_t* q_full = pv_done + 1;
  uint64_t* o_full = q_full + 1;
  uint64_t* drain = o_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  float* red = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + C::kBarBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = p.group;
  const int QP = 128 / G;           // query positions per tile
  const int rows_valid = QP * G;    // rows that carry a (position, head)
  const int n_qblocks = (int)((p.n + QP - 1) / QP);
  const int qb = n_qblocks - 1 - (int)blockIdx.x;  // longest rows first
  const int h = blockIdx.y;
  const int b = blockIdx.z;
  const PrefillUnit& u = p.u[h];
  const int64_t t0 = p.t0;
  const int64_t p0 = t0 + (int64_t)qb * QP;
  const int64_t p_last = min(p0 + QP, t0 + p.n) - 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], C::kSoftmaxWarps);  // one arrival per softmax warp
    }
    mbar_init(p_full, C::kSoftmaxWarps);
    mbar_init(pv_done, 1);
    mbar_init(q_full, 1);
    mbar_init(o_full, 1);
    mbar_init(drain, 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  KeySeq<BN> seq;
  seq.init(u, t0, p.n, p0, p_last);
  bool aborted = false;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      prefetch_tensormap(&q_map);
      prefetch_tensormap(&ck_map);
      prefetch_tensormap(&cv_map);
      prefetch_tensormap(&ring_map);
      mbar_arrive_expect_tx(q_full, (uint32_t)(C::kSlabs * rows_valid * 128));
      const int32_t qrow = (int32_t)((int64_t)b * p.n + (int64_t)qb * QP);
#pragma unroll
      for (int sl = 0; sl < C::kSlabs; ++sl)
        tma_load_3d(sQ + sl * C::kQSlab, &q_map, sl * 64, h * G, qrow, q_full);
      const int64_t krow0 = u.k_row0 + (int64_t)(p.row0 + b) * u.stride;
      const int64_t vrow0 = u.v_row0 + (int64_t)(p.row0 + b) * u.stride;
      // two walks of the same key sequence: K tiles run one tile ahead of V tiles
      KeySeq<BN> seq_v = seq;
      uint32_t it_k = 0, it_v = 0;
      auto issue = [&](KeySeq<BN>& sq, uint32_t& it, uint64_t* full, uint64_t* empty,
                       uint8_t* buf, int64_t row0, const CUtensorMap* cmap) -> bool {
        int hist;
        int64_t j0;
        if (!sq.next(hist, j0)) return false;
        const int s = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1u;
        if (wait_or_abort(&empty[s], ph ^ 1u, p.err, aborted)) {
          uint8_t* d = buf + s * C::kTileBytes;
          mbar_arrive_expect_tx(&full[s], C::kTileBytes);
#pragma unroll
          for (int sl = 0; sl < C::kSlabs; ++sl) {
#pragma unroll
            for (int hf = 0; hf < BN / 64; ++hf) {
              const uint32_t off = sl * C::kKVSlab + hf * 64 * 128;
              if (hist)
                tma_load_2d(d + off, &ring_map, sl * 64, (int32_t)(row0 + j0 + hf * 64), &full[s]);
              else
                tma_load_3d(d + off, cmap, sl * 64, h, (int32_t)((int64_t)b * p.n + j0 + hf * 64),
                            &full[s]);
            }
          }
        }
        ++it;
        return true;
      };
      bool more_k = issue(seq, it_k, k_full, k_empty, sK, krow0, &ck_map);
      while (true) {
        if (more_k) more_k = issue(seq, it_k, k_full, k_empty, sK, krow0, &ck_map);
        if (!issue(seq_v, it_v, v_full, v_empty, sV, vrow0, &cv_map)) break;
      }
      // every issued copy has landed before shared memory can go away
      bool late = false;
      for (uint32_t j = it_k > (uint32_t)STAGES ? it_k - STAGES : 0u; j < it_k; ++j)
        wait_or_abort(&k_full[j % STAGES], (j / STAGES) & 1u, p.err, late);
      for (uint32_t j = it_v > (uint32_t)STAGES ? it_v - STAGES : 0u; j < it_v; ++j)
        wait_or_abort(&v_full[j % STAGES], (j / STAGES) & 1u, p.err, late);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------- mma issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(128, BN, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, true);
      const uint32_t tO = tmem + C::kColO;
      const uint32_t tP = tmem + C::kColP;
      const uint32_t q_base = smem_u32(sQ);
      wait_or_abort(q_full, 0, p.err, aborted);
      auto issue_pv = [&](uint32_t jj) {
        bool ok = wait_or_abort(p_full, jj & 1u, p.err, aborted);
        ok = ok && wait_or_abort(&v_full[jj % STAGES], (jj / STAGES) & 1u, p.err, aborted);
        if (ok) {
          tc_fence_after();
          const uint32_t v_base = smem_u32(sV + (jj % STAGES) * C::kTileBytes);
#pragma unroll
          for (int kk = 0; kk < BN / 16; ++kk) {  // 16 keys = 8 packed P columns
            const uint64_t bd = smem_desc_sw128(v_base + kk * 2048, C::kKVSlab, 1024);
            umma_bf16_tmem_a(tO, tP + kk * 8, bd, idesc_pv, (jj > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(pv_done);
          umma_commit(&v_empty[jj % STAGES]);
        }
      };
      uint32_t j = 0;
      int hist;
      int64_t j0;
      while (seq.next(hist, j0)) {
        const int s = j % STAGES;
        const int sb = j % SBUF;
        bool ok = wait_or_abort(&k_full[s], (j / STAGES) & 1u, p.err, aborted);
        ok = ok && wait_or_abort(&s_free[sb], ((j / SBUF) & 1u) ^ 1u, p.err, aborted);
        if (ok) {
          tc_fence_after();
          const uint32_t k_base = smem_u32(sK + s * C::kTileBytes);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint64_t a = smem_desc_sw128(q_base + (kk >> 2) * C::kQSlab + (kk & 3) * 32, 16, 1024);
            const uint64_t bd = smem_desc_sw128(k_base + (kk >> 2) * C::kKVSlab + (kk & 3) * 32, 16, 1024);
            umma_bf16(tmem + sb * BN, a, bd, idesc_qk, kk > 0 ? 1u : 0u);
          }
          umma_commit(&s_full[sb]);
          umma_commit(&k_empty[s]);  // the K tile is free once its QK^T has read it
        }
        if (j >= 1) issue_pv(j - 1);
        ++j;
      }
      if (j >= 1) issue_pv(j - 1);
      if (!aborted) umma_commit(o_full);
      // every mma issued has finished before TMEM is released
      umma_commit(drain);
      bool late = false;
      wait_or_abort(drain, 0, p.err, late);
    }
  } else {
    // ---------------------------------------------------------------- softmax
    const int quarter = warp & 3;        // TMEM lanes this warp may access
    const int half = (warp - 2) >> 2;     // which share of the columns (SPLIT = 2)
    const int r = quarter * 32 + lane;
    const int cbase = half * C::kCW;      // first S column of this warp
    const int obase = half * C::kOW;      // first O column of this warp
    const int64_t pr = p0 + r / G;
    const bool row_ok = r < rows_valid && pr <= p_last;
    const int qh = h * G + r % G;
    const int64_t W = u.window;
    const int64_t lo_r = W == 0 ? 0 : (pr - W + 1 > 0 ? pr - W + 1 : 0);  // first visible key
    const uint32_t t_lane = tmem + ((uint32_t)(quarter * 32) << 16);
    const float c = p.scale_log2;
    float m_used = -INFINITY, l = 0.f;  // running max (log2 units) and sum of weights
    uint32_t j = 0;
    int hist;
    int64_t j0;
    auto clampi = [](int64_t v) -> int { return (int)(v < -1 ? -1 : (v > BN + 1 ? BN + 1 : v)); };
    while (seq.next(hist, j0)) {
      const int sb = j % SBUF;
      // columns e of this tile visible to row pr: [a0, b0) U [a1, b1)
      int a0 = 0, b0 = 0, a1 = 0, b1 = 0;
      if (row_ok) {
        if (hist == 0) {  // chunk keys at positions t0 + j0 + e, held while j0 + e < n
          const int64_t hi = min(pr - t0 - j0, p.n - 1 - j0);  // causal, held
          a0 = clampi(lo_r - t0 - j0);
          b0 = clampi(hi + 1);
          b1 = clampi(min(seq.S - t0 - j0, hi + 1));  // chunk keys that are sinks
        } else if (hist == 2) {  // sink slots: slot j holds position j, always visible
          b0 = clampi(seq.n_sink - j0);
        } else {
          // window region, slots relative to its start: position S + v in slot
          // S + (v mod Wr) for the region's v-th held token
          const int64_t jw = j0 - seq.S, lo_v = lo_r - seq.S;
          if (seq.tw <= seq.Wr) {  // not yet wrapped
            a0 = clampi(lo_v - jw);
            b0 = clampi(seq.n_win - jw);
          } else {  // wrapped: slots < r0 hold the newest run, slots >= r0 the older one
            const int64_t A = lo_v - seq.tw + seq.r0;  // first visible slot of the newest run
            a0 = clampi(A - jw);
            b0 = clampi(seq.r0 - jw);
            a1 = clampi(A + seq.Wr - jw);
            b1 = clampi(seq.Wr - jw);
          }
        }
      }
      const bool full_vis = (a0 <= 0 && b0 >= BN) || (a1 <= 0 && b1 >= BN);
      const bool warp_full = __all_sync(0xffffffffu, full_vis);  // warp-uniform fast path
      if (warp_wait_or_abort(&s_full[sb], (j / SBUF) & 1u, p.err, aborted)) tc_fence_after();
      // this warp's S columns, read once into registers; the S buffer is then free
      // for the QK^T of tile j + 2 while this tile's softmax runs
      uint32_t sv[C::kCW];
#pragma unroll
      for (int cc = 0; cc < C::kCW / 32; ++cc)
        tmem_ld32(t_lane + sb * BN + cbase + cc * 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[cc * 32]));
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[sb]);
      // row max of the visible logits (raw; scale > 0 so max(z) c = max(z c))
      float mx;
      {
        float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
        if (warp_full) {
#pragma unroll
          for (int e = 0; e < C::kCW; ++e) m4[e & 3] = fmaxf(m4[e & 3], __uint_as_float(sv[e]));
        } else {
#pragma unroll
          for (int e = 0; e < C::kCW; ++e) {
            const int col = cbase + e;
            const bool vis = full_vis || (col >= a0 && col < b0) || (col >= a1 && col < b1);
            if (!vis) sv[e] = __float_as_uint(-INFINITY);
            m4[e & 3] = fmaxf(m4[e & 3], __uint_as_float(sv[e]));
          }
        }
        mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
        if (SPLIT > 1) {  // combine with the warp holding the other columns of these rows
          float* rb = red + (j & 1) * 256;
          rb[half * 128 + r] = mx;
          asm volatile("bar.sync %0, 64;" ::"r"(1 + quarter) : "memory");
          mx = fmaxf(mx, rb[(1 - half) * 128 + r]);
        }
        mx *= c;
      }
      const float m_new = fmaxf(m_used, mx);
      const bool resc = m_new - m_used > 8.f;  // false while both are -inf
      float alpha = 1.f;
      if (resc) {
        alpha = ex2(m_used - m_new);
        m_used = m_new;
        l *= alpha;
      }
      const float bias = m_used == -INFINITY ? 0.f : m_used;

      // weights 2^(z c - m), computed in place (masked logits are -inf: weight 0);
      // the exponent arguments and the row sum in packed fp32 pairs
      float2 s2a = make_float2(0.f, 0.f), s2b = make_float2(0.f, 0.f);
      {
        const float2 c2 = make_float2(c, c), nb2 = make_float2(-bias, -bias);
#pragma unroll
        for (int e = 0; e < C::kCW; e += 2) {
          const float2 y = fma2(make_float2(__uint_as_float(sv[e]), __uint_as_float(sv[e + 1])), c2, nb2);
          const float2 w = make_float2(ex2(y.x), ex2(y.y));
          if (e & 2) s2b = add2(s2b, w); else s2a = add2(s2a, w);
          sv[e] = __float_as_uint(w.x);
          sv[e + 1] = __float_as_uint(w.y);
        }
      }
      float s4[4] = {s2a.x, s2a.y, s2b.x, s2b.y};
      const float sum = (s4[0] + s4[1]) + (s4[2] + s4[3]);

      // PV of the previous tile has read P and added into O: only now may P be
      // overwritten and O rescaled (rare: the reference max only moves when a
      // row's max grows by more than 2^8)
      if (j >= 1 && warp_wait_or_abort(pv_done, (j - 1) & 1u, p.err, aborted)) tc_fence_after();
      if (j >= 1 && __any_sync(0xffffffffu, resc)) {
        const uint32_t tO = t_lane + C::kColO + obase;
#pragma unroll
        for (int cc = 0; cc < C::kOW / 32; ++cc) {
          uint32_t rr[32];
          tmem_ld32(tO + cc * 32, rr);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) rr[e] = __float_as_uint(__uint_as_float(rr[e]) * alpha);
          tmem_st32(tO + cc * 32, rr);
        }
        tmem_st_wait();
      }
      // P row -> TMEM as bf16 pairs (A operand of the PV mma, read from tensor memory)
      {
        uint32_t pk[C::kCW / 2];
#pragma unroll
        for (int e = 0; e < C::kCW / 2; ++e)
          pk[e] = pack_bf16(__uint_as_float(sv[2 * e]), __uint_as_float(sv[2 * e + 1]));
        const uint32_t tPw = t_lane + C::kColP + (cbase >> 1);
        if constexpr (C::kCW / 2 == 16) {
          tmem_st16(tPw, *reinterpret_cast<const uint32_t(*)[16]>(pk));
        } else {
#pragma unroll
          for (int cc = 0; cc < C::kCW / 64; ++cc)
            tmem_st32(tPw + cc * 32, *reinterpret_cast<const uint32_t(*)[32]>(&pk[cc * 32]));
        }
        tmem_st_wait();
      }
      l += sum;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);  // P rows written (and O rescaled)
      ++j;
    }
    // epilogue: O / l for this row
    if (warp_wait_or_abort(o_full, 0, p.err, aborted)) tc_fence_after();
    if (SPLIT > 1) {  // each warp of the pair summed only its columns
      red[half * 128 + r] = l;  // every max exchange was read before o_full
      asm volatile("bar.sync %0, 64;" ::"r"(1 + quarter) : "memory");
      l += red[(1 - half) * 128 + r];
    }
    const float inv = l > 0.f ? 1.f / l : 0.f;
    float* dst = p.out + (((int64_t)b * p.n + (pr - t0)) * p.n_q_heads + qh) * D + obase;
#pragma unroll
    for (int cc = 0; cc < C::kOW / 32; ++cc) {
      uint32_t rr[32];
      tmem_ld32(t_lane + C::kColO + obase + cc * 32, rr);
      tmem_ld_wait();
      if (row_ok) {
#pragma unroll
        for (int e = 0; e < 32; e += 4)
          *reinterpret_cast<float4*>(dst + cc * 32 + e) =
              make_float4(__uint_as_float(rr[e]) * inv, __uint_as_float(rr[e + 1]) * inv,
                          __uint_as_float(rr[e + 2]) * inv, __uint_as_float(rr[e + 3]) * inv);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
}

template <int D, int BN, int STAGES, int SPLIT, int SBUF = 2, int CTAS = 1>
static cudaError_t launch_tc(const PrefillParams& p, const CUtensorMap& qm, const CUtensorMap& km,
                             const CUtensorMap& vm, const CUtensorMap& rm, cudaStream_t s) {
  using C = TcCfg<D, BN, STAGES, SPLIT, SBUF, CTAS>;
  cudaError_t e = cudaFuncSetAttribute(prefill_tc_kernel<D, BN, STAGES, SPLIT, SBUF, CTAS>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
  if (e != cudaSuccess) return e;
  const int QP = 128 / p.group;
  dim3 grid((unsigned)((p.n + QP - 1) / QP), (unsigned)p.n_units, (unsigned)p.batch);
  prefill_tc_kernel<D, BN, STAGES, SPLIT, SBUF, CTAS><<<grid, C::kThreads, C::kSmem, s>>>(qm, km, vm, rm, p);
  return cudaGetLastError();
}

int prefill_tc_rows_per_tile(int group) { return (128 / group) * group; }

cudaError_t launch_prefill_tc(const PrefillParams& p, int head_dim, const CUtensorMap& q_map,
                              const CUtensorMap& ck_map, const CUtensorMap& cv_map,
                              const CUtensorMap& ring_map, cudaStream_t s) {
  if (p.n == 0) return cudaSuccess;
  switch (head_dim) {
    case 64: return launch_tc<64, 64, 3, 1, 1, 2>(p, q_map, ck_map, cv_map, ring_map, s);
    case 128: return launch_tc<128, 64, 2, 1, 1, 2>(p, q_map, ck_map, cv_map, ring_map, s);
    case 256: return launch_tc<256, 64, 2, 1>(p, q_map, ck_map, cv_map, ring_map, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace hwkv
