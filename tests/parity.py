"""Teacher-forced parity of the CUDA path against the CPU oracle.

For every checked frame the oracle starts from the GPU's pre-frame state
(slot order converted to position order), runs the same bf16 inputs, and the
two results are compared:

* attention output: max |O_gpu - O_oracle| <= 2e-2 (bf16 inputs, fp32
  accumulation on the GPU);
* importance: |g - o| <= 1e-3 |o| + 1e-6 per pool member (state columns mapped
  through the pre-frame slot positions);
* selection: with tau the oracle's B-th best score, every candidate whose
  score lies outside [tau (1 - 1e-3), tau (1 + 1e-3)] gets the same keep /
  evict decision; the kept count is min(B, pool); kept positions are unique;
* state rows are bit copies of the rows of the frame that produced them;
* decode cache rows are bit copies of every frame's K and V.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import torch

import oracle
from paper_2605_31598_gb300 import StateKV, make_config
from paper_2605_31598_gb300.inputs import batch_qkv

OUT_ATOL = 2e-2
IMP_RTOL = 1e-3
IMP_ATOL = 1e-6
BAND = 1e-3


def _bits(t):
    return oracle.as_bf16_bits(t)


def _oracle_frames(lays, pre, units, q, k, v):
    """The oracle's frame for every unit, teacher-forced from the GPU's
    pre-frame state ``pre[unit]``; units run on host threads side by side
    (the C loops run outside the Python lock)."""
    bits = {u: (_bits(q[u[0], u[1]]), _bits(k[u[0], u[1]]), _bits(v[u[0], u[1]])) for u in units}

    def one(u):
        count, ppos, pk, pv, vlen = pre[u]
        lay = lays[u]
        lay.set_state(np.full(lay.n_kv, count, np.int32), ppos, pk, pv, vlen)
        return lay.prefill_frame(*bits[u])

    workers = max(1, min(len(units), os.cpu_count() or 1))
    with ThreadPoolExecutor(max_workers=workers) as ex:
        return dict(zip(units, ex.map(one, units)))


def run_parity(shape, nframes, *, kind=None, seed=0, check_frames=None, causal=True,
               units=None, call_layers=None, want_importance=True, host_api=False,
               stats=None, selection=0):
    """Run ``nframes`` frames on the GPU; compare the frames in ``check_frames``.

    units: (stream, layer) pairs to compare (default: all).  call_layers:
    split each frame into calls over these layer ranges [(begin, count), ...].
    selection: 0 the per-KV-head top-B (Eq. 6), 2 the layer-level top-B
    (App. A), whose ranking score is the importance summed over the KV heads
    and whose kept positions must agree across heads.
    Returns the StateKV engine (for extra checks by the caller).
    """
    S, L = shape.num_streams, shape.num_layers
    T, Hq, Hkv, d, B = (shape.tokens_per_frame, shape.num_q_heads, shape.num_kv_heads,
                        shape.head_dim, shape.state_capacity)
    G = Hq // Hkv
    eng = StateKV(make_config(shape, causal=causal, host_staging=host_api, selection=selection))
    units = units or [(s, l) for s in range(S) for l in range(L)]
    check_frames = set(range(1, nframes + 1) if check_frames is None else check_frames)
    call_layers = call_layers or [(0, L)]
    hist_k = {u: [] for u in units}
    hist_v = {u: [] for u in units}
    lays = {u: oracle.OracleLayer(Hq, Hkv, d, T, B, shape.max_frames, causal=causal,
                                  policy=selection)
            for u in units}
    stats = stats if stats is not None else {}
    stats.setdefault("max_out_err", 0.0)
    stats.setdefault("max_imp_rel", 0.0)
    stats.setdefault("band_candidates", 0)
    stats.setdefault("decisions", 0)
    for n in range(1, nframes + 1):
        q, k, v = batch_qkv(shape, n, streams=range(S), layers=range(L), seed=seed,
                            device="cuda", kind=kind)
        out = torch.full_like(q, float("nan"))
        imp = (torch.full((S, L, Hkv, B + T), float("nan"), device="cuda")
               if want_importance else None)
        checking = n in check_frames
        pre = {}
        if checking:
            torch.cuda.synchronize()
            for u in units:
                kk, vv, pp, info = eng.state(*u)
                pre[u] = (info.count, pp.cpu().numpy().astype(np.int64), _bits(kk), _bits(vv),
                          info.virtual_len)
        for (lb, lc) in call_layers:
            sl = slice(lb, lb + lc)
            qs, ks, vs, os_ = (x[:, sl].contiguous() for x in (q, k, v, out))
            imps = imp[:, sl].contiguous() if imp is not None else None
            if host_api:
                qh, kh, vh = (x.cpu().pin_memory() for x in (qs, ks, vs))
                oh = torch.empty_like(os_, device="cpu").pin_memory()
                ih = torch.empty_like(imps, device="cpu").pin_memory() if imps is not None else None
                rc = eng.prefill_frame_host(qh, kh, vh, oh, ih, layer_begin=lb, layer_count=lc)
                assert rc == 0, f"frame {n}: statekv_prefill_frame_host returned {rc}"
                torch.cuda.synchronize()
                os_.copy_(oh)
                if imps is not None:
                    imps.copy_(ih)
            else:
                rc = eng.prefill_frame(qs, ks, vs, os_, imps, layer_begin=lb, layer_count=lc)
                assert rc == 0, f"frame {n}: statekv_prefill_frame returned {rc}"
            out[:, sl] = os_
            if imp is not None:
                imp[:, sl] = imps
        torch.cuda.synchronize()
        for u in units:
            s, l = u
            hist_k[u].append(_bits(k[s, l]))
            hist_v[u].append(_bits(v[s, l]))
        if not checking:
            continue
        refs = _oracle_frames(lays, pre, units, q, k, v)
        for u in units:
            s, l = u
            count, ppos, pk, pv, vlen = pre[u]
            o_ref, imp_ref, kept_ref = refs[u]
            o_gpu = out[s, l].float().cpu().numpy()
            err = float(np.abs(o_gpu - o_ref).max())
            stats["max_out_err"] = max(stats["max_out_err"], err)
            assert err <= OUT_ATOL, f"frame {n} unit {u}: max |dO| = {err}"
            kk, vv, pp, info = eng.state(s, l)
            post_pos = pp.cpu().numpy()
            post_k, post_v = _bits(kk), _bits(vv)
            allk = np.concatenate(hist_k[u])  # [n*T][Hkv][d]
            allv = np.concatenate(hist_v[u])
            rank_score = imp_ref.sum(axis=0) if selection == 2 else None  # layer level
            if selection == 2:
                heads = [sorted(post_pos[h][post_pos[h] >= 0].tolist()) for h in range(Hkv)]
                assert all(x == heads[0] for x in heads), f"frame {n} unit {u}: heads disagree"
            for h in range(Hkv):
                # importance: map GPU slot j -> oracle column (position order)
                order = {int(p): i for i, p in enumerate(np.sort(ppos[h, :count]))}
                if imp is not None:
                    g = imp[s, l, h].cpu().numpy().astype(np.float64)
                    o_cols = np.zeros(B + T)
                    for j in range(count):
                        o_cols[j] = imp_ref[h, order[int(ppos[h, j])]]
                    o_cols[B:] = imp_ref[h, B:]
                    assert np.all(g[count:B] == 0), f"frame {n} unit {u}: empty slots not 0"
                    dif = np.abs(g[:count] - o_cols[:count])
                    ok_s = dif <= IMP_RTOL * np.abs(o_cols[:count]) + IMP_ATOL
                    dif_f = np.abs(g[B:] - o_cols[B:])
                    ok_f = dif_f <= IMP_RTOL * np.abs(o_cols[B:]) + IMP_ATOL
                    assert ok_s.all() and ok_f.all(), (
                        f"frame {n} unit {u} head {h}: importance mismatch "
                        f"(state worst {dif.max() if count else 0}, frame worst {dif_f.max()})")
                    rel = np.concatenate([dif / np.maximum(np.abs(o_cols[:count]), 1e-30),
                                          dif_f / np.maximum(np.abs(o_cols[B:]), 1e-30)])
                    stats["max_imp_rel"] = max(stats["max_imp_rel"], float(rel.max()))
                # selection outside the tolerance band
                gpos = post_pos[h][post_pos[h] >= 0]
                assert len(gpos) == min(B, count + T), f"frame {n} unit {u}: count {len(gpos)}"
                assert len(set(gpos.tolist())) == len(gpos), f"frame {n} unit {u}: duplicate"
                gset = set(int(x) for x in gpos)
                cand_pos = np.concatenate([np.sort(ppos[h, :count]), vlen + np.arange(T)])
                rs = imp_ref[h] if rank_score is None else rank_score
                cand_score = np.concatenate([rs[:count], rs[B:]])
                cand_kept = np.concatenate([kept_ref[h, :count], kept_ref[h, B:]]).astype(bool)
                if count + T > B and B > 0:
                    tau = np.sort(cand_score)[::-1][B - 1]
                    outside = np.abs(cand_score - tau) > BAND * tau
                else:
                    outside = np.ones(len(cand_pos), bool)
                gk = np.array([int(p) in gset for p in cand_pos])
                stats["band_candidates"] += int((~outside).sum())
                stats["decisions"] += len(cand_pos)
                bad = outside & (gk != cand_kept)
                assert not bad.any(), (f"frame {n} unit {u} head {h}: selection differs "
                                       f"outside the band at positions {cand_pos[bad][:8]}")
                # state rows are bit copies of their source rows
                valid = post_pos[h] >= 0
                src = post_pos[h][valid]
                assert np.array_equal(post_k[h][valid], allk[src, h]), f"frame {n}: state K"
                assert np.array_equal(post_v[h][valid], allv[src, h]), f"frame {n}: state V"
            # decode cache holds every frame so far
            ck, cv, cinfo = eng.cache(s, l)
            Ln = n * T
            assert cinfo.length == Ln
            assert np.array_equal(_bits(ck[:, :Ln]), allk.transpose(1, 0, 2)), f"frame {n}: cache K"
            assert np.array_equal(_bits(cv[:, :Ln]), allv.transpose(1, 0, 2)), f"frame {n}: cache V"
    assert eng.sync() == 0
    return eng


def run_free_running(shape, nframes, *, kind=None, seed=0, stats=None):
    """Free-running parity of one (stream, layer): the oracle keeps its own
    state from frame 1 on and is never reset to the GPU's.

    Until the first near-tie at the selection boundary both sides must hold
    the same state (as position sets) after every frame, with outputs and
    importance within the tolerances above.  A frame is a near-tie when the
    B-th and (B+1)-th best oracle scores are within 2e-3 of each other
    (relative): each may move by the 1e-3 importance tolerance, so either
    decision is correct there and the two runs may part.  The run stops after
    that frame.  Returns the number of frames compared and the frame of the
    first near-tie (None when there was none).
    """
    T, Hq, Hkv, d, B = (shape.tokens_per_frame, shape.num_q_heads, shape.num_kv_heads,
                        shape.head_dim, shape.state_capacity)
    assert shape.num_streams == 1 and shape.num_layers == 1
    eng = StateKV(make_config(shape))
    lay = oracle.OracleLayer(Hq, Hkv, d, T, B, shape.max_frames)
    stats = stats if stats is not None else {}
    tie_frame = None
    n = 0
    for n in range(1, nframes + 1):
        q, k, v = batch_qkv(shape, n, streams=[0], layers=[0], seed=seed, device="cuda", kind=kind)
        torch.cuda.synchronize()
        _, _, gpre, ginfo = eng.state(0, 0)
        gpre = gpre.cpu().numpy().astype(np.int64)
        count = int(ginfo.count)
        opre = [lay.state_positions(h) for h in range(Hkv)]
        for h in range(Hkv):
            assert sorted(gpre[h, :count].tolist()) == opre[h].tolist(), \
                f"frame {n} head {h}: states parted before a near-tie"
        out = torch.full_like(q, float("nan"))
        imp = torch.full((1, 1, Hkv, B + T), float("nan"), device="cuda")
        assert eng.prefill_frame(q, k, v, out, imp) == 0
        o_ref, imp_ref, kept_ref = lay.prefill_frame(_bits(q[0, 0]), _bits(k[0, 0]), _bits(v[0, 0]))
        torch.cuda.synchronize()
        err = float(np.abs(out[0, 0].float().cpu().numpy() - o_ref).max())
        assert err <= OUT_ATOL, f"frame {n}: max |dO| = {err}"
        g_imp = imp[0, 0].cpu().numpy().astype(np.float64)
        _, _, gpost, _ = eng.state(0, 0)
        gpost = gpost.cpu().numpy()
        near_tie = False
        for h in range(Hkv):
            col = {int(p): i for i, p in enumerate(opre[h])}
            o_cols = np.zeros(B + T)
            for j in range(count):
                o_cols[j] = imp_ref[h, col[int(gpre[h, j])]]
            o_cols[B:] = imp_ref[h, B:]
            sel = np.r_[0:count, B:B + T]
            assert np.all(np.abs(g_imp[h, sel] - o_cols[sel]) <= IMP_RTOL * np.abs(o_cols[sel]) + IMP_ATOL), \
                f"frame {n} head {h}: importance"
            scores = np.sort(np.concatenate([imp_ref[h, :count], imp_ref[h, B:]]))[::-1]
            if B > 0 and len(scores) > B:
                tau = scores[B - 1]
                near_tie |= bool(scores[B - 1] - scores[B] <= 2 * BAND * tau)
        if near_tie:
            tie_frame = n
            break
        for h in range(Hkv):
            gset = sorted(int(x) for x in gpost[h] if x >= 0)
            assert gset == lay.state_positions(h).tolist(), f"frame {n} head {h}: kept sets differ"
    assert eng.sync() == 0
    stats["frames"] = n
    stats["first_near_tie"] = tie_frame
    return n, tie_frame
