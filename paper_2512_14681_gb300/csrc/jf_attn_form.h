// Launch form of the split-KV attention (host side; no CUDA types, so that the rule compiles and is
// tested on the host alone).
//
// A unit (chain, KV head, tile of 128 query rows) runs on 8 CTAs, one key lane each. The clustered
// form makes them an 8-CTA cluster and folds the lane states in parallel after a cluster barrier,
// but only `max_clusters` such clusters are resident at once (15 on a GB300: 120 of 152 SMs). The
// unclustered form can use every SM, and the last lane of a unit folds all its rows. Both fold in
// lane order with the same arithmetic, so the choice affects time only.
#pragma once

namespace jf {

// Units of a forward of M rows spread evenly over `chains` chains (exact for equal chains, e.g.
// B sequences with one n-row window each), capped by the launch's upper bound.
inline int attn_units_estimate(int M, int chains, int units_bound, int Hkv, int G, int q_rows_per_tile) {
  const int cb = chains > 0 ? chains : 1;
  const long long rows_per_chain = (M + cb - 1) / cb;
  const long long tiles = (rows_per_chain * G + q_rows_per_tile - 1) / q_rows_per_tile;
  const long long est = (long long)Hkv * cb * tiles;
  return est < units_bound ? (int)est : units_bound;
}

// true: the clustered form, which is taken unless the unclustered one needs fewer waves of units
// (ties go to the clustered form, whose parallel fold is faster).
inline bool attn_use_clusters(int units, int lanes, int max_clusters, int num_sms) {
  const int mc = max_clusters > 0 ? max_clusters : 1;
  const int waves_clustered = (units + mc - 1) / mc;
  const int waves_unclustered = (int)(((long long)units * lanes + num_sms - 1) / num_sms);
  return waves_clustered <= waves_unclustered;
}

}  // namespace jf
