"""Host logic of the layer-1 bit-row backward's schedule (no GPU): the
degree order of layer 1's nodes and layer 2's CSR map built in that order's
sequence, as `pipeline.Network` prepares them, and the bit-row byte
accounting of the benchmark for a batch that is not a whole number of
1024-sample blocks."""
import numpy as np

import paper_2602_07400_gb300 as bl
from paper_2602_07400_gb300 import synth
from paper_2602_07400_gb300.pipeline import Network


def test_network_orders_layer1_by_consumer_count_with_a_matching_csr_map():
    wl = synth.Workload("t", 64, 20, 4, 1.0, [64, 128, 192], (300, 200), 6, 10.0)
    conn1, th1, conn2, th2 = synth.network(wl, seed=4)
    net = Network(conn1, th1, conn2, th2, wl.w_in, device="cpu")
    order = net.order1.numpy()
    off, edge = (t.numpy() for t in (net.off2, net.edge2))
    offo, edgeo, poso = (t.numpy() for t in (net.off2o, net.edge2o, net.pos2o))
    deg = np.diff(off)
    assert sorted(order.tolist()) == list(range(net.w1))          # a permutation
    assert np.all(np.diff(deg[order]) <= 0)                         # heaviest first
    for p in range(net.w1):                                        # ties by index
        if p and deg[order[p]] == deg[order[p - 1]]:
            assert order[p] > order[p - 1]
    # position p of the ordered map holds node order[p]'s edges, in the
    # same increasing order as the map by node (so the terms sum alike)
    for p, j in enumerate(order):
        np.testing.assert_array_equal(edgeo[offo[p]:offo[p + 1]], edge[off[j]:off[j + 1]])
    # pos2o places every edge at its position in the ordered map
    np.testing.assert_array_equal(edgeo[poso], np.arange(edgeo.size))
    # every edge e = j2 * k2 + slot of the ordered map reads node conn2[j2][slot]
    for p, j in enumerate(order):
        for e in edgeo[offo[p]:offo[p + 1]]:
            assert conn2.reshape(-1)[e] == j


def test_bit_row_accounting_pads_the_batch_to_whole_blocks():
    import bench
    wl = synth.WORKLOADS["mnist"]
    B = 1000                       # one partly filled 1024-sample block
    work = bench.call_work(wl, B, fuse_dy1=True, bytes1=True, bits1=True)
    xw1 = 4 * wl.w_in * 32
    assert work["encode"][0] == B * wl.d + xw1
    assert work["forward1"][0] - xw1 == bench.call_work(wl, B, fuse_dy1=True, bytes1=True)["forward1"][0] - wl.w_in * B
    assert bl.bitrow_words(B) == 32 and bl.bitrow_words(1024) == 32 and bl.bitrow_words(1025) == 64
    assert bl.bitrow_words(0) == 0
