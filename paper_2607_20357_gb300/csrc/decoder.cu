// Device-side schedule of the gated decoder (Sec. 3.2) and the row kernels
// around the GEMMs: RMSNorm, final norm of the last rows, RoPE table.
//
// For every layer l the schedule kernel turns the gates into work lists, so
// that gated-off work is never issued and the host never learns k or T:
//  * e_{b,l,j} = (l < P) or (layer_gate[b,l] and group_gate[b,l,j]);
//  * consecutive samples with the same non-zero group mask form one row
//    segment (samples with mask 0 skip the layer: residual bypass);
//  * QKV tiles cover only the Q/K/V columns of active groups, gate/up tiles
//    only active FFN channels. These N-sparse lists are built per group, over
//    maximal runs of consecutive samples in which that group runs (other
//    groups' bits do not cut a run), and adjacent groups whose on/off pattern
//    over the samples is the same share one column block; so mixed masks do
//    not fragment the row tiles, and all-on batches get the segment tiles;
//  * O and down tiles carry the segment mask so their K loop visits only
//    active groups' rows of W_O / W_down;
//  * attention items are (sample, active head, block of kAttnQ queries).
#include "kernels.cuh"

namespace svl {

constexpr int kMaxNT = 512;

struct NTile {
  int n0, ncols, mat;
};

// Column runs of consecutive active groups, cut into tiles of `step`.
SVL_DEVINL int build_runs(NTile* out, int cnt, int mask, int G, int width, int step, int mat) {
  int j = 0;
  while (j < G) {
    if (!((mask >> j) & 1)) { ++j; continue; }
    int j1 = j;
    while (j1 + 1 < G && ((mask >> (j1 + 1)) & 1)) ++j1;
    const int c0 = j * width, c1 = (j1 + 1) * width;
    for (int n0 = c0; n0 < c1 && cnt < kMaxNT; n0 += step) out[cnt++] = {n0, min(step, c1 - n0), mat};
    j = j1 + 1;
  }
  return cnt;
}

// Emits mt x nt tiles of one segment in raster bands. mband > 0: bands of
// `mband` m-tiles, each sweeping all n-tiles while its input rows stay in L2
// (the tiles of one n-tile follow each other, so concurrent CTAs share its
// weights too). Otherwise bands of `nband` n-tiles, each sweeping all m-tiles
// while its weight columns stay in L2.
__device__ void emit_tiles(int4* tiles, int base, int cap, int r0, int r1, const NTile* nt, int n_nt, int kmask,
                           uint32_t* status, int bm = kBM_SCHED, int nband = kNBand, int mband = 0) {
  const int mt = (r1 - r0 + bm - 1) / bm;
  const int total = mt * n_nt;
  for (int t = threadIdx.x; t < total; t += blockDim.x) {
    int mi, ni;
    if (mband > 0) {
      const int band = t / (mband * n_nt);
      const int rem = t - band * mband * n_nt;
      const int bh = min(mband, mt - band * mband);
      ni = rem / bh;
      mi = band * mband + rem % bh;
    } else {
      const int band = t / (mt * nband);
      const int rem = t - band * mt * nband;
      const int bw = min(nband, n_nt - band * nband);
      mi = rem / bw;
      ni = band * nband + rem % bw;
    }
    const int m0 = r0 + mi * bm;
    const int idx = base + t;
    if (idx >= cap) {
      report(status, SVL_DEV_BAD_INDEX);
      continue;
    }
    const NTile n = nt[ni];
    tiles[idx] = make_int4(m0, min(m0 + bm, r1), n.n0, n.ncols | (n.mat << 16) | (kmask << 24));
  }
}

// The persistent GEMM runs tiles in waves of num_sms. When the last wave is
// at most half full, each of its tiles is cut into two half-width tiles
// (which then still fit in one wave and finish in about half the time).
// `head` > 0: halves must hold whole heads of that width (RoPE epilogue).
// Called by the whole block once the list is complete; the appended halves
// keep the order of their tiles (a ballot prefix over the eligible ones).
// s_scan: blockDim.x / 32 ints of shared memory. Returns the new count.
__device__ int split_tail(int4* tiles, int count, int cap, int num_sms, int head, int* s_scan) {
  const int r = count % num_sms;
  if (r == 0 || 2 * r > num_sms) return count;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int eligible = 0;  // in the chunks before this one
  for (int c0 = count - r; c0 < count; c0 += blockDim.x) {
    const int i = c0 + static_cast<int>(threadIdx.x);
    int4 t = make_int4(0, 0, 0, 0);
    bool e = false;
    if (i < count) {
      t = tiles[i];
      const int nc = t.w & 0xFFFF, half = nc / 2;
      e = nc >= 64 && !(half & 15) && !(head > 0 && half % head);
    }
    const unsigned bal = __ballot_sync(0xffffffffu, e);
    if (lane == 0) s_scan[warp] = __popc(bal);
    __syncthreads();
    int before = eligible + __popc(bal & ((1u << lane) - 1u)), chunk = 0;
    for (int w = 0; w < nw; ++w) {
      if (w < warp) before += s_scan[w];
      chunk += s_scan[w];
    }
    __syncthreads();  // s_scan is reused by the next chunk
    if (e && count + before < cap) {
      const int nc = t.w & 0xFFFF, half = nc / 2;
      tiles[i] = make_int4(t.x, t.y, t.z, (t.w & ~0xFFFF) | half);
      tiles[count + before] = make_int4(t.x, t.y, t.z + half, (t.w & ~0xFFFF) | (nc - half));
    }
    eligible += chunk;
  }
  return count + min(eligible, cap - count);
}

// Residual GEMMs (O, down) cut the tiles of a last wave that is at most half
// full along K instead: each of the r tail tiles is repeated s times (s =
// num_sms / r, at most 8, within the list capacity and the partial buffer),
// the copies compute shares of the tile's K blocks side by side in that wave
// and the last to finish sums them. Full-width tiles keep the tensor core's
// widest MMAs. Called by the whole block once the list is complete; thread 0
// writes {first copy index, r, s} to info. Returns the count.
__device__ int split_k_tail(int4* tiles, int count, int cap, int num_sms, int units, int* info) {
  const int sp = ksplit_shares(count, cap, num_sms, units);
  const int r = sp < 2 ? 0 : count % num_sms;
  const int first = count - r;
  if (threadIdx.x == 0) {
    info[0] = first;
    info[1] = r;
    info[2] = sp < 2 ? 1 : sp;
  }
  if (sp < 2) return count;
  // copy `part` (1 .. sp-1) of tail tile i goes to count + (part - 1) r + i
  for (int idx = threadIdx.x; idx < r * (sp - 1); idx += blockDim.x) tiles[count + idx] = tiles[first + idx % r];
  return count + r * (sp - 1);
}

// Shared-memory copies of the layer's per-sample inputs: row offsets
// cu[0..B] and the effective group mask of every sample (bit j: group j
// runs). Filled by the whole block, so the serial walks below read shared
// memory only.
struct SchedShared {
  int* cu;
  uint8_t* mask;
};

SVL_DEVINL bool group_on(const SchedShared& sh, int b, int j) { return (sh.mask[b] >> j) & 1; }

// Emits the tiles of an N-sparse GEMM list of layer l: for each block of
// adjacent groups with the same on/off pattern over the non-empty samples,
// the maximal row runs of samples where the block runs, times the block's
// columns (`cols(j0, j1, nt)` fills the n-tiles). Returns the tile count.
// Called by the whole block; thread 0 walks groups and samples.
template <class Cols>
__device__ int emit_group_runs(const ScheduleArgs& a, const SchedShared& sh, int4* tiles, int cap, NTile* nt,
                               int* s_nnt, int* s_run, Cols cols) {
  const int tid = threadIdx.x, B = a.B, G = a.G;
  int off = 0;
  int j0 = 0;
  while (j0 < G) {
    // the block [j0, j1]: following groups with the same pattern
    if (tid == 0) {
      int j1 = j0;
      for (; j1 + 1 < G; ++j1) {
        bool same = true;
        for (int b = 0; b < B && same; ++b)
          if (sh.cu[b + 1] > sh.cu[b]) same = group_on(sh, b, j1 + 1) == group_on(sh, b, j0);
        if (!same) break;
      }
      s_run[2] = j1;
      *s_nnt = cols(j0, j1, nt);
      s_run[3] = 0;  // next sample to look at
    }
    __syncthreads();
    const int j1 = s_run[2];
    while (true) {
      if (tid == 0) {
        // next maximal run of non-empty samples (empty ones are transparent) where the block runs
        int b = s_run[3], r0 = -1, r1 = -1;
        for (; b < B; ++b) {
          const int q0 = sh.cu[b], q1 = sh.cu[b + 1];
          if (q1 <= q0) continue;
          if (group_on(sh, b, j0)) {
            if (r0 < 0) r0 = q0;
            r1 = q1;
          } else if (r0 >= 0) {
            break;
          }
        }
        s_run[0] = r0;
        s_run[1] = r1;
        s_run[3] = b;
      }
      __syncthreads();
      const int r0 = s_run[0], r1 = s_run[1];
      if (r0 < 0) break;
      emit_tiles(tiles, off, cap, r0, r1, nt, *s_nnt, 0, a.status, a.nsparse_rows, 0, a.mband);
      off += ((r1 - r0 + a.nsparse_rows - 1) / a.nsparse_rows) * *s_nnt;
      __syncthreads();
    }
    j0 = j1 + 1;
    __syncthreads();
  }
  return min(off, cap);
}

__global__ void __launch_bounds__(256) schedule_kernel(ScheduleArgs a) {
  __shared__ NTile nt[kMaxNT];
  __shared__ int s_nseg, s_nnt;
  __shared__ int s_heads[256];
  __shared__ int s_run[4];
  __shared__ int s_scan[8];  // per-warp counts of split_tail (256 threads)
  pdl_trigger();
  pdl_wait();
  extern __shared__ int sched_dyn[];
  const int l = blockIdx.x, tid = threadIdx.x;
  const int B = a.B, G = a.G;
  int4* seg = a.seg + static_cast<size_t>(l) * B;
  uint8_t* act = a.act + static_cast<size_t>(l) * B;
  const SchedShared sh{sched_dyn, reinterpret_cast<uint8_t*>(sched_dyn + B + 1)};
  for (int b = tid; b <= B; b += blockDim.x) sh.cu[b] = a.cu_seqlens[b];
  for (int b = tid; b < B; b += blockDim.x) {
    int mask = 0;
    for (int j = 0; j < G; ++j) {
      const bool e = (l < a.P) || (a.layer_gate[b * a.L + l] && a.group_gate[(b * a.L + l) * G + j]);
      mask |= e ? (1 << j) : 0;
    }
    sh.mask[b] = static_cast<uint8_t>(mask);
  }
  __syncthreads();

  if (tid == 0) {
    int ns = 0;
    for (int b = 0; b < B; ++b) {
      const int mask = sh.mask[b];
      const int r0 = sh.cu[b], r1 = sh.cu[b + 1];
      act[b] = (mask != 0 && r1 > r0) ? 1 : 0;
      if (mask == 0 || r1 <= r0) continue;
      if (ns > 0 && seg[ns - 1].z == mask && seg[ns - 1].y == r0) {
        seg[ns - 1].y = r1;
      } else {
        seg[ns] = make_int4(r0, r1, mask, 0);
        ++ns;
      }
    }
    s_nseg = ns;
  }
  __syncthreads();
  const int nseg = s_nseg;
  const int hq = (a.A / G) * a.dh, hk = (a.Akv / G) * a.dh;

  // ---- QKV (N-sparse over active groups' Q, K, V columns, per group block)
  auto qkv_cols = [&](int j0, int j1, NTile* out) {
    const int mask = ((1 << (j1 + 1)) - 1) & ~((1 << j0) - 1);
    int c = build_runs(out, 0, mask, G, hq, 256, 0);
    c = build_runs(out, c, mask, G, hk, 256, 1);
    return build_runs(out, c, mask, G, hk, 256, 2);
  };
  int off = emit_group_runs(a, sh, a.qkv_tiles + static_cast<size_t>(l) * a.qkv_cap, a.qkv_cap, nt, &s_nnt, s_run,
                            qkv_cols);
  __syncthreads();
  off = split_tail(a.qkv_tiles + static_cast<size_t>(l) * a.qkv_cap, off, a.qkv_cap, a.nsparse_wave, a.dh, s_scan);
  if (tid == 0) a.qkv_count[l] = off;

  // ---- O projection (K-sparse: kmask = segment mask), all D columns
  off = 0;
  if (tid == 0) s_nnt = build_runs(nt, 0, 1, 1, a.D, 256, 0);
  __syncthreads();
  for (int s = 0; s < nseg; ++s) {
    const int4 sg = seg[s];
    emit_tiles(a.o_tiles + static_cast<size_t>(l) * a.o_cap, off, a.o_cap, sg.x, sg.y, nt, s_nnt, sg.z, a.status,
               kBM_SCHED, kNBandO);
    off += ((sg.y - sg.x + kBM_SCHED - 1) / kBM_SCHED) * s_nnt;
  }
  __syncthreads();
  off = split_k_tail(a.o_tiles + static_cast<size_t>(l) * a.o_cap, min(off, a.o_cap), a.o_cap, a.num_sms, a.ks_units,
                     a.ks_info + static_cast<size_t>(l) * 8);
  if (tid == 0) a.o_count[l] = off;
  // ---- down projection: same tiles shape as O
  off = 0;
  for (int s = 0; s < nseg; ++s) {
    const int4 sg = seg[s];
    emit_tiles(a.dn_tiles + static_cast<size_t>(l) * a.dn_cap, off, a.dn_cap, sg.x, sg.y, nt, s_nnt, sg.z, a.status);
    off += ((sg.y - sg.x + kBM_SCHED - 1) / kBM_SCHED) * s_nnt;
  }
  __syncthreads();
  off = split_k_tail(a.dn_tiles + static_cast<size_t>(l) * a.dn_cap, min(off, a.dn_cap), a.dn_cap, a.num_sms,
                     a.ks_units, a.ks_info + static_cast<size_t>(l) * 8 + 4);
  if (tid == 0) a.dn_count[l] = off;
  __syncthreads();

  // ---- gate/up (N-sparse over active FFN channels, 128 per tile, per group block)
  auto gu_cols = [&](int j0, int j1, NTile* out) {
    const int mask = ((1 << (j1 + 1)) - 1) & ~((1 << j0) - 1);
    return build_runs(out, 0, mask, G, a.Di / G, 128, 0);
  };
  off = emit_group_runs(a, sh, a.gu_tiles + static_cast<size_t>(l) * a.gu_cap, a.gu_cap, nt, &s_nnt, s_run, gu_cols);
  __syncthreads();
  if (tid == 0) a.gu_count[l] = off;

  // ---- attention items: per active sample and active head, blocks of kAttnQ
  // queries, latest first (the kernel takes units from the front of the list,
  // so one head's blocks run at about the same time and share its keys in L2)
  off = 0;
  int4* items = a.attn_items + static_cast<size_t>(l) * a.attn_cap;
  const int hpg = a.A / G;
  for (int s = 0; s < nseg; ++s) {
    const int4 sg = seg[s];
    if (tid == 0) {
      int nh = 0;
      for (int j = 0; j < G; ++j)
        if ((sg.z >> j) & 1)
          for (int h = 0; h < hpg && nh < 256; ++h) s_heads[nh++] = j * hpg + h;
      s_nnt = nh;
    }
    __syncthreads();
    const int nh = s_nnt;
    // samples inside the segment
    int lo = 0, hi = B;
    while (hi - lo > 1) {  // first sample of the segment
      const int mid = (lo + hi) >> 1;
      if (sh.cu[mid] <= sg.x) lo = mid; else hi = mid;
    }
    for (int b = lo; b < B && sh.cu[b] < sg.y; ++b) {
      const int r0 = sh.cu[b], r1 = sh.cu[b + 1];
      if (r1 <= r0) continue;
      const int nq = (r1 - r0 + kAttnQ - 1) / kAttnQ;
      const int total = nq * nh;
      for (int t = tid; t < total; t += blockDim.x) {
        const int qi = nq - 1 - t % nq;
        const int h = s_heads[t / nq];
        const int q0 = r0 + qi * kAttnQ;
        const int idx = off + t;
        if (idx < a.attn_cap) items[idx] = make_int4(q0, min(q0 + kAttnQ, r1), r0, h);
        else report(a.status, SVL_DEV_BAD_INDEX);
      }
      off += total;
    }
    __syncthreads();
  }
  if (tid == 0) {
    a.attn_count[l] = min(off, a.attn_cap);
    a.attn_next[l] = 0;
  }
}

void launch_schedule(const ScheduleArgs& a, cudaStream_t s) {
  launch_pdl(schedule_kernel, a.L, 256, static_cast<size_t>(a.B + 1) * sizeof(int) + a.B, s, a);
}

// LLM-side compute controller (Sec. 3.2), one block per sample:
//   h~ = h_b^(P) + W_k2 SiLU(W_k1 PE(kappa))          (Eq. 7; h_b^(P) = the budget
//                                                     token's row after P layers)
//   logit[l - P][j] = W_h[(l - P) G + j] . h~ + c_h    (gate head)
//   group (l, j) runs if l < P or logit > 0 (sigma > 0.5; no noise at inference)
// With `project` and b < 1, the token count being committed, the fewest
// active groups of layers >= P are switched off, lowest logit first (equal
// logits: lower l * G + j first), until Eq. 8 at S = S_text + k is within
// b * C_full (Sec. 3.3 "Inference").
constexpr int kCtlThreads = 256;
__global__ void __launch_bounds__(kCtlThreads) controller_kernel(CtlArgs a) {
  extern __shared__ float ctl_smem[];
  float* ht = ctl_smem;           // [D] fused state
  float* lg = ctl_smem + a.D;     // [(L - P) * G] gate logits
  __shared__ double pe[256], hid[256];
  __shared__ int keep_groups;
  __shared__ long long n_on_sh;
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int L = a.L, G = a.G, P = min(a.P, a.L), H = a.H, D = a.D;
  const int ng = (L - P) * G;
  const int row = a.cu_seqlens[b + 1] - 1;
  // e_kappa = W_k2 SiLU(W_k1 PE(kappa)), PE as Eq. 5
  if (tid < H) {
    const int half = H / 2, f = tid < half ? tid : tid - half;
    const double arg = 1000.0 * static_cast<double>(a.kappa[b]) * pow(10000.0, -2.0 * f / H);
    pe[tid] = tid < half ? sin(arg) : cos(arg);
  }
  if (tid == 0) {
    keep_groups = -1;
    n_on_sh = 0;
  }
  __syncthreads();
  if (tid < H) {
    double s = 0.0;
    for (int j = 0; j < H; ++j) s += static_cast<double>(__bfloat162float(a.kap_w1[tid * H + j])) * pe[j];
    hid[tid] = s / (1.0 + exp(-s));
  }
  __syncthreads();
  for (int d = tid; d < D; d += blockDim.x) {
    double s = row >= 0 ? static_cast<double>(__bfloat162float(a.X[static_cast<size_t>(row) * D + d])) : 0.0;
    for (int j = 0; j < H; ++j) s += static_cast<double>(__bfloat162float(a.kap_w2[static_cast<size_t>(d) * H + j])) * hid[j];
    ht[d] = static_cast<float>(s);
  }
  __syncthreads();
  // gate head: one warp per logit, lanes along D
  for (int o = warp; o < ng; o += blockDim.x / 32) {
    const __nv_bfloat16* wr = a.gate_w + static_cast<size_t>(o) * D;
    float acc = 0.f;
    for (int d = lane; d < D; d += 32) acc = fmaf(__bfloat162float(wr[d]), ht[d], acc);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (lane == 0) {
      lg[o] = acc + a.gate_c[o];
      if (a.gate_logits) a.gate_logits[static_cast<size_t>(b) * ng + o] = lg[o];
    }
  }
  __syncthreads();
  // raw gates and their count (prefix groups always on)
  int on = 0;
  for (int idx = tid; idx < L * G; idx += blockDim.x) on += (idx < P * G || lg[idx - P * G] > 0.f) ? 1 : 0;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) on += __shfl_xor_sync(0xffffffffu, on, off);
  if (lane == 0 && on) atomicAdd(reinterpret_cast<unsigned long long*>(&n_on_sh), static_cast<unsigned long long>(on));
  __syncthreads();
  uint32_t flags = 0;
  int drop = 0;
  if (a.project && a.budget[b] < 1.0f) {
    const long long D64 = D, Dkv = a.Dkv, Di = a.Di, V = a.V, G64 = G, L64 = L;
    const long long lin = 4 * D64 * D64 + 4 * D64 * Dkv + 6 * D64 * Di;
    const long long nv = a.vis_off[b + 1] - a.vis_off[b], st = a.text_len[b];
    const long long S_full = nv + st, S = st + a.k[b];
    const long long c_full = G64 * L64 * (lin * S_full + 4 * D64 * S_full * S_full) + G64 * 2 * D64 * V * S_full;
    const double limit = static_cast<double>(a.budget[b]) * static_cast<double>(c_full);
    const long long per = lin * S + 4 * D64 * S * S, lm = G64 * 2 * D64 * V * S;
    const long long n_on = n_on_sh, n_min = static_cast<long long>(P) * G;
    if (static_cast<double>(n_on * per + lm) > limit) {
      for (long long nk = n_min + tid; nk < n_on; nk += blockDim.x)
        if (static_cast<double>(nk * per + lm) <= limit) atomicMax(&keep_groups, static_cast<int>(nk));
      __syncthreads();
      if (n_on > n_min) flags |= SVL_FLAG_GROUPS_DROPPED;
      if (keep_groups < 0) flags |= SVL_FLAG_OVER_BUDGET;
      drop = static_cast<int>(n_on - (keep_groups < 0 ? n_min : keep_groups));
    }
  }
  uint8_t* go = a.group_gate + static_cast<size_t>(b) * L * G;
  for (int idx = tid; idx < L * G; idx += blockDim.x) {
    bool active = idx < P * G || lg[idx - P * G] > 0.f;
    if (active && drop > 0 && idx >= P * G) {
      const float v = lg[idx - P * G];
      int rank = 0;
      for (int j = P * G; j < L * G; ++j) {
        const float w = lg[j - P * G];
        if (w > 0.f && (w < v || (w == v && j < idx))) ++rank;
      }
      active = rank >= drop;
    }
    go[idx] = active ? 1 : 0;
  }
  __syncthreads();
  for (int l = tid; l < L; l += blockDim.x) {
    int any = 0;
    for (int j = 0; j < G; ++j) any |= go[l * G + j];
    a.layer_gate[static_cast<size_t>(b) * L + l] = any ? 1 : 0;
  }
  if (tid == 0 && a.flags) a.flags[b] |= flags;
}

void launch_controller(const CtlArgs& a, cudaStream_t s) {
  const size_t smem = sizeof(float) * (static_cast<size_t>(a.D) + static_cast<size_t>(a.L - min(a.P, a.L)) * a.G);
  static bool configured = false;
  if (!configured && smem > 48 * 1024) {
    cudaFuncSetAttribute(controller_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
    configured = true;
  }
  launch_pdl(controller_kernel, a.B, kCtlThreads, smem, s, a);
}

// ---------------------------------------------------------------- RMSNorm

SVL_DEVINL void norm_row(const __nv_bfloat16* x, const __nv_bfloat16* g, __nv_bfloat16* y, int D, float eps,
                         int lane) {
  const uint4* xv = reinterpret_cast<const uint4*>(x);
  const uint4* gv = reinterpret_cast<const uint4*>(g);
  uint4* yv = reinterpret_cast<uint4*>(y);
  float ss = 0.f;
  for (int c = lane; c < D / 8; c += 32) {
    const uint4 u = xv[c];
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = unpack_bf16x2(w[i]);
      ss += f.x * f.x + f.y * f.y;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float inv = rsqrtf(ss / static_cast<float>(D) + eps);
  for (int c = lane; c < D / 8; c += 32) {
    const uint4 u = xv[c], gg = gv[c];
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
    const uint32_t q[4] = {gg.x, gg.y, gg.z, gg.w};
    uint32_t o[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = unpack_bf16x2(w[i]), h = unpack_bf16x2(q[i]);
      o[i] = pack_bf16x2(f.x * inv * h.x, f.y * inv * h.y);
    }
    yv[c] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

__global__ void rmsnorm_kernel(NormArgs a) {
  pdl_trigger();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp;
  const int T = a.cu_seqlens[a.B];
  if (r >= T || r >= a.t_cap) return;
  if (a.act && !a.act[find_sample(a.cu_seqlens, a.B, r)]) return;
  norm_row(a.X + static_cast<size_t>(r) * a.D, a.gain, a.Y + static_cast<size_t>(r) * a.D, a.D, a.eps, lane);
}

__global__ void final_rows_kernel(NormArgs a, int n_pad) {
  pdl_trigger();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * (blockDim.x >> 5) + warp;
  if (b >= n_pad) return;
  __nv_bfloat16* y = a.Y + static_cast<size_t>(b) * a.D;
  const int r1 = b < a.B ? a.cu_seqlens[b + 1] : 0, r0 = b < a.B ? a.cu_seqlens[b] : 0;
  if (b >= a.B || r1 <= r0) {
    for (int c = lane; c < a.D / 8; c += 32) reinterpret_cast<uint4*>(y)[c] = make_uint4(0, 0, 0, 0);
    return;
  }
  norm_row(a.X + static_cast<size_t>(r1 - 1) * a.D, a.gain, y, a.D, a.eps, lane);
}

// Sum of squares of every packed row of X into slot 0 of ss ([slots][ss_ld]),
// the other slots zeroed: the first layer's fused RMSNorm reads these.
__global__ void norm_init_kernel(const __nv_bfloat16* X, const int* cu_seqlens, int B, int t_cap, int D, float* ss,
                                 int ss_ld, int slots) {
  pdl_trigger();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp;
  if (r >= cu_seqlens[B] || r >= t_cap) return;
  const uint4* xv = reinterpret_cast<const uint4*>(X + static_cast<size_t>(r) * D);
  float acc = 0.f;
  for (int c = lane; c < D / 8; c += 32) {
    const uint4 u = xv[c];
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = unpack_bf16x2(w[i]);
      acc = fmaf(f.x, f.x, fmaf(f.y, f.y, acc));
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  for (int i = lane; i < slots; i += 32) ss[static_cast<size_t>(i) * ss_ld + r] = i == 0 ? acc : 0.f;
}

void launch_norm_init(const __nv_bfloat16* X, const int* cu_seqlens, int B, int t_cap, int D, float* ss, int ss_ld,
                      int slots, cudaStream_t s) {
  const int grid = (t_cap + 7) / 8;
  if (grid > 0) launch_pdl(norm_init_kernel, grid, 256, 0, s, X, cu_seqlens, B, t_cap, D, ss, ss_ld, slots);
}

// W'[r][c] = W[r][c] * g[c] (a norm gain folded into the projection after it)
__global__ void fold_gain_kernel(const __nv_bfloat16* W, const __nv_bfloat16* g, __nv_bfloat16* out, int64_t rows,
                                 int cols) {
  const int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (i >= rows * cols) return;
  const int c = static_cast<int>(i % cols);
  out[i] = __float2bfloat16_rn(__bfloat162float(W[i]) * __bfloat162float(g[c]));
}

// flag = 0 unless every gain is exactly 1
__global__ void gain_is_one_kernel(const __nv_bfloat16* g, int n, int* flag) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
    if (__bfloat162float(g[i]) != 1.f) *flag = 0;
}

cudaError_t fold_gain(const __nv_bfloat16* W, const __nv_bfloat16* g, __nv_bfloat16* out, int64_t rows, int cols,
                      cudaStream_t s) {
  const int64_t n = rows * cols;
  fold_gain_kernel<<<static_cast<unsigned>((n + 255) / 256), 256, 0, s>>>(W, g, out, rows, cols);
  return cudaGetLastError();
}

cudaError_t gain_is_one(const __nv_bfloat16* g, int n, int* flag, cudaStream_t s) {
  gain_is_one_kernel<<<(n + 255) / 256, 256, 0, s>>>(g, n, flag);
  return cudaGetLastError();
}

void launch_rmsnorm(const NormArgs& a, cudaStream_t s) {
  const int grid = (a.t_cap + 7) / 8;
  if (grid > 0) launch_pdl(rmsnorm_kernel, grid, 256, 0, s, a);
}

void launch_final_last_rows(const NormArgs& a, int n_pad, cudaStream_t s) {
  launch_pdl(final_rows_kernel, (n_pad + 7) / 8, 256, 0, s, a, n_pad);
}

__global__ void selftest_wait_kernel(uint32_t* status, long long cycles) {
  __shared__ uint64_t bar;
  __shared__ int abort;
  if (threadIdx.x == 0) {
    abort = 0;
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !mbar_wait(&bar, 0, &abort, cycles)) report(status, SVL_DEV_TIMEOUT);
}

void launch_selftest_wait(uint32_t* status, long long cycles, cudaStream_t s) {
  selftest_wait_kernel<<<1, 32, 0, s>>>(status, cycles);
}

__global__ void rope_table_kernel(float2* cs, int max_seq, int dh, double theta) {
  const int half = dh / 2;
  const long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  if (i >= static_cast<long long>(max_seq) * half) return;
  const int f = static_cast<int>(i / max_seq), p = static_cast<int>(i % max_seq);
  const double ang = static_cast<double>(p) * pow(theta, -2.0 * f / dh);
  cs[i] = make_float2(static_cast<float>(cos(ang)), static_cast<float>(sin(ang)));
}

void launch_rope_table(float2* cs, int max_seq, int dh, double theta, cudaStream_t s) {
  const long long n = static_cast<long long>(max_seq) * (dh / 2);
  rope_table_kernel<<<static_cast<int>((n + 255) / 256), 256, 0, s>>>(cs, max_seq, dh, theta);
}

}  // namespace svl
